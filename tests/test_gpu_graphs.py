"""Graph replay of plain forwards: repeated zsaa_forward calls (eager, then
captured, then replayed) give bit-identical logits and kept positions, also
on the legacy default stream and after switching replay off."""

import pytest
import torch

from paper_2509_01190_gb300 import inputs as I
from tests.helpers import need_gpu

pytestmark = pytest.mark.gpu

SHAPE = I.ModelShape("graph-bf16", 3, 256, 4, 2, 64, 512, 1008)


def test_graph_replay_is_bit_identical(zlib):
    need_gpu()
    z = zlib
    B, L = 3, 200
    weights = I.make_weights(SHAPE, device="cuda")
    model = z.Model(z.config_from_shape(SHAPE), weights, B, L)
    tok = torch.from_numpy(I.make_tokens(B, L, SHAPE.vocab)).cuda()
    for accel in (1.0, 3.0):
        sched, _ = z.zsaa_plan(model, L, accel)
        outs = []
        for stream in (torch.cuda.Stream(), torch.cuda.default_stream()):
            logits = torch.empty(B, sched[-1], SHAPE.vocab, device="cuda")
            kept = torch.empty(B, sched[-1], device="cuda", dtype=torch.int32)
            with torch.cuda.stream(stream):
                for _ in range(4):  # eager, capture, replay, replay
                    logits.fill_(float("nan"))
                    z.zsaa_forward(model, tok, B, L, accel, logits, kept, stream=stream)
                    stream.synchronize()
                    outs.append((logits.clone(), kept.clone()))
        z.zsaa_model_set_graphs(model, False)
        logits = torch.empty(B, sched[-1], SHAPE.vocab, device="cuda")
        kept = torch.empty(B, sched[-1], device="cuda", dtype=torch.int32)
        z.zsaa_forward(model, tok, B, L, accel, logits, kept)
        z.zsaa_sync(model)
        z.zsaa_model_set_graphs(model, True)
        for lg, kp in outs:
            assert torch.equal(lg, logits) and torch.equal(kp, kept)
