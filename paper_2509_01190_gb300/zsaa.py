"""Python binding of libzsaa.so (ctypes; argument marshalling only).

Every function here has the name of a C entry point in ``include/zsaa.h`` and
forwards to it: torch tensors become raw device pointers (``data_ptr()``), and
a non-OK status becomes a ``ZsaaError``.  No step of the computation runs in
Python.  If the library has not been built, ``lib()`` raises; there is no
fallback implementation.
"""

from __future__ import annotations

import ctypes as C
import os
from typing import Dict, List, Optional, Sequence, Tuple

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "lib", "libzsaa.so")

ZSAA_OK, ZSAA_ERR_INVALID_ARG, ZSAA_ERR_OOM, ZSAA_ERR_CUDA, ZSAA_ERR_TIMEOUT, ZSAA_ERR_UNSUPPORTED = range(6)
ZSAA_F32, ZSAA_BF16 = 0, 1
ZSAA_SCORE_SOFTSCORE_VNORM, ZSAA_SCORE_SOFTSCORE = 0, 1
ZSAA_PLAN_COST, ZSAA_PLAN_RATE = 0, 1
ZSAA_FLAG_FORCE_KEEP_LAST = 1
EPI_STORE, EPI_RESID, EPI_SWIGLU, EPI_STORE_F32, EPI_ROPE = range(5)

EXPORTED = [
    "zsaa_plan_config", "zsaa_model_create", "zsaa_model_destroy", "zsaa_plan", "zsaa_forward",
    "zsaa_forward_ex", "zsaa_forward_host", "zsaa_score_select", "zsaa_score_select_ex",
    "zsaa_op_linear", "zsaa_op_attention", "zsaa_op_colmass", "zsaa_sync", "zsaa_device_status",
    "zsaa_last_error", "zsaa_version", "zsaa_trace_begin", "zsaa_trace_end",
    "zsaa_score_select_noalloc", "zsaa_model_set_graphs", "zsaa_cache_create", "zsaa_cache_destroy",
    "zsaa_prefill", "zsaa_decode_step", "zsaa_cache_layer", "zsaa_cache_bytes",
    "zsaa_op_attention_ex", "zsaa_op_colmass_ex", "zsaa_plan_varlen_config", "zsaa_plan_varlen",
    "zsaa_forward_varlen", "zsaa_forward_masked", "zsaa_forward_marked", "zsaa_selftest_wait_timeout",
    "zsaa_gemm_schedule",
]


class ZsaaError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"zsaa status {status}: {msg}")
        self.status = status


class zsaa_config(C.Structure):
    _fields_ = [
        ("n_layers", C.c_int), ("d_model", C.c_int), ("n_heads", C.c_int), ("n_kv_heads", C.c_int),
        ("head_dim", C.c_int), ("ffn_dim", C.c_int), ("vocab", C.c_int), ("n_classes", C.c_int),
        ("rope_theta", C.c_float), ("rms_eps", C.c_float), ("dtype", C.c_int), ("tau", C.c_int),
        ("prune_mask", C.c_uint64), ("force_keep_last", C.c_int), ("score_mode", C.c_int),
        ("plan_mode", C.c_int), ("bidirectional", C.c_int),
    ]


class zsaa_weights(C.Structure):
    _fields_ = [("embed", C.c_void_p), ("layers", C.POINTER(C.c_void_p)),
                ("final_norm", C.c_void_p), ("head", C.c_void_p)]


class zsaa_forward_opts(C.Structure):
    _fields_ = [("forced_idx", C.c_void_p), ("scores_out", C.c_void_p), ("idx_out", C.c_void_p),
                ("hidden_out", C.c_void_p), ("n_layers_run", C.c_int), ("hidden_in", C.c_void_p),
                ("pos_in", C.c_void_p), ("first_layer", C.c_int), ("plan_L", C.c_int)]


class zsaa_trace_row(C.Structure):
    _fields_ = [("name", C.c_char * 32), ("launches", C.c_int), ("ms", C.c_double),
                ("flops", C.c_double), ("bytes", C.c_double)]


_LIB = None

_P = C.c_void_p
_I = C.c_int
_D = C.c_double


def lib():
    """Load libzsaa.so (once).  Raises if it is missing."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run `python -m paper_2509_01190_gb300.build`")
        L = C.CDLL(LIB_PATH)
        sig = {
            "zsaa_plan_config": ([C.POINTER(zsaa_config), _I, _D, C.POINTER(_I), C.POINTER(_D)], _I),
            "zsaa_model_create": ([C.POINTER(zsaa_config), C.POINTER(zsaa_weights), _I, _I, C.POINTER(_P)], _I),
            "zsaa_model_destroy": ([_P], None),
            "zsaa_plan": ([_P, _I, _D, C.POINTER(_I), C.POINTER(_D)], _I),
            "zsaa_forward": ([_P, _P, _I, _I, _D, _P, _P, _P], _I),
            "zsaa_forward_ex": ([_P, _P, _I, _I, _D, _P, _P, C.POINTER(zsaa_forward_opts), _P], _I),
            "zsaa_forward_host": ([_P, _P, _I, _I, _D, _P, _P, _P], _I),
            "zsaa_score_select": ([_P, _I, _I, _I, _I, _P, _P, _P], _I),
            "zsaa_score_select_ex": ([_P, _I, _I, _I, _I, _I, _I, _P, _P, _P, _P, _P], _I),
            "zsaa_score_select_noalloc": ([_P, _I, _I, _I, _I, _P, _P, _P], _I),
            "zsaa_model_set_graphs": ([_P, _I], _I),
            "zsaa_op_linear": ([_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P, _I, _I, C.c_float, _P], _I),
            "zsaa_gemm_schedule": ([_I, _I, _I, _I, _I, _I, _I, _I, _P, _P, C.c_int64, C.POINTER(C.c_int64)], _I),
            "zsaa_op_attention": ([_P, _I, _I, _I, _I, _I, _I, _P, _P, _P], _I),
            "zsaa_op_colmass": ([_P, _P, _I, _I, _I, _I, _I, _I, _P, _P], _I),
            "zsaa_op_attention_ex": ([_P, _I, _I, _I, _I, _I, _I, _I, _P, _P, _P], _I),
            "zsaa_plan_varlen_config": ([C.POINTER(zsaa_config), _P, _I, _D, C.POINTER(_I), C.POINTER(_D)], _I),
            "zsaa_plan_varlen": ([_P, _P, _I, _D, C.POINTER(_I), C.POINTER(_D)], _I),
            "zsaa_forward_varlen": ([_P, _P, _P, _I, _D, _P, _P, C.POINTER(zsaa_forward_opts), _P], _I),
            "zsaa_forward_masked": ([_P, _P, _I, _I, _D, _P, _P, C.POINTER(zsaa_forward_opts), _P], _I),
            "zsaa_forward_marked": ([_P, _P, _I, _I, _D, _P, _P, C.POINTER(zsaa_forward_opts), _P], _I),
            "zsaa_op_colmass_ex": ([_P, _P, _I, _I, _I, _I, _I, _I, _I, _P, _P], _I),
            "zsaa_sync": ([_P, _P], _I),
            "zsaa_device_status": ([], _I),
            "zsaa_selftest_wait_timeout": ([_P], _I),
            "zsaa_last_error": ([], C.c_char_p),
            "zsaa_version": ([], C.c_char_p),
            "zsaa_trace_begin": ([_P], _I),
            "zsaa_trace_end": ([_P, C.POINTER(zsaa_trace_row), _I, C.POINTER(_I)], _I),
            "zsaa_cache_create": ([_P, _I, _I, _D, _I, C.POINTER(_P)], _I),
            "zsaa_cache_destroy": ([_P], None),
            "zsaa_prefill": ([_P, _P, _P, _P, C.POINTER(zsaa_forward_opts), _P], _I),
            "zsaa_decode_step": ([_P, _P, _P, _P, _P], _I),
            "zsaa_cache_layer": ([_P, _I, C.POINTER(_P), C.POINTER(_P), C.POINTER(_P), C.POINTER(_I),
                                  C.POINTER(_I), C.POINTER(_I)], _I),
            "zsaa_cache_bytes": ([_P, C.POINTER(C.c_size_t), C.POINTER(C.c_size_t)], _I),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _LIB = L
    return _LIB


def _check(st: int):
    if st != ZSAA_OK:
        raise ZsaaError(st, lib().zsaa_last_error().decode())


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ------------------------------------------------------------------ config

def make_config(n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn_dim, vocab, n_classes=0,
                rope_theta=500000.0, rms_eps=1e-5, dtype="bf16", tau=5,
                prune_layers: Sequence[int] = (), force_keep_last=True,
                score_mode="softscore_vnorm", plan_mode="cost", bidirectional=False) -> zsaa_config:
    mask = 0
    for layer in prune_layers:
        mask |= 1 << (int(layer) - 1)
    return zsaa_config(
        n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn_dim, vocab, n_classes,
        float(rope_theta), float(rms_eps), ZSAA_BF16 if dtype == "bf16" else ZSAA_F32, tau, mask,
        1 if force_keep_last else 0,
        ZSAA_SCORE_SOFTSCORE_VNORM if score_mode == "softscore_vnorm" else ZSAA_SCORE_SOFTSCORE,
        ZSAA_PLAN_COST if plan_mode == "cost" else ZSAA_PLAN_RATE, 1 if bidirectional else 0)


def config_from_shape(shape, prune_layers: Optional[Sequence[int]] = None, **overrides) -> zsaa_config:
    """zsaa_config from any object with the ModelShape attributes."""
    kw = dict(n_layers=shape.n_layers, d_model=shape.d_model, n_heads=shape.n_heads,
              n_kv_heads=shape.n_kv_heads, head_dim=shape.head_dim, ffn_dim=shape.ffn_dim,
              vocab=shape.vocab, n_classes=shape.n_classes, rope_theta=shape.rope_theta,
              rms_eps=shape.rms_eps, dtype=shape.dtype,
              prune_layers=shape.prune_layers() if prune_layers is None else prune_layers,
              plan_mode=shape.plan_mode, bidirectional=getattr(shape, "bidirectional", False),
              score_mode=getattr(shape, "score_mode", "softscore_vnorm"))
    kw.update(overrides)
    return make_config(**kw)


# ------------------------------------------------------------------ planner

def zsaa_plan_config(cfg: zsaa_config, L: int, accel: float) -> Tuple[List[int], float]:
    sched = (C.c_int * (cfg.n_layers + 1))()
    alpha = C.c_double()
    _check(lib().zsaa_plan_config(C.byref(cfg), L, float(accel), sched, C.byref(alpha)))
    return list(sched), alpha.value


# ------------------------------------------------------------------ model

LAYER_SLOTS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd")


class Model:
    """Owns a zsaa_model handle and keeps the borrowed weight tensors alive."""

    def __init__(self, cfg: zsaa_config, weights: Dict, max_B: int, max_L: int):
        self.cfg = cfg
        self._weights = weights
        ptrs = []
        for lw in weights["layers"]:
            ptrs += [lw[k].data_ptr() for k in LAYER_SLOTS]
        self._layer_ptrs = (C.c_void_p * len(ptrs))(*ptrs)
        w = zsaa_weights(weights["embed"].data_ptr(), self._layer_ptrs,
                         weights["final_norm"].data_ptr(), weights["head"].data_ptr())
        h = C.c_void_p()
        _check(lib().zsaa_model_create(C.byref(cfg), C.byref(w), max_B, max_L, C.byref(h)))
        self.handle = h
        self.max_B, self.max_L = max_B, max_L

    def close(self):
        if getattr(self, "handle", None) is not None and self.handle.value:
            lib().zsaa_model_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def zsaa_model_create(cfg: zsaa_config, weights: Dict, max_B: int, max_L: int) -> Model:
    return Model(cfg, weights, max_B, max_L)


def zsaa_model_destroy(model: Model):
    model.close()


def zsaa_model_set_graphs(model: Model, enable: bool):
    _check(lib().zsaa_model_set_graphs(model.handle, 1 if enable else 0))


def zsaa_plan(model: Model, L: int, accel: float) -> Tuple[List[int], float]:
    sched = (C.c_int * (model.cfg.n_layers + 1))()
    alpha = C.c_double()
    _check(lib().zsaa_plan(model.handle, L, float(accel), sched, C.byref(alpha)))
    return list(sched), alpha.value


def zsaa_forward(model: Model, token_ids, B: int, L: int, accel: float, logits_out,
                 kept_pos_out=None, stream=None):
    _check(lib().zsaa_forward(model.handle, _ptr(token_ids), B, L, float(accel), _ptr(logits_out),
                              _ptr(kept_pos_out), _stream(stream)))


def zsaa_forward_ex(model: Model, token_ids, B: int, L: int, accel: float, logits_out,
                    kept_pos_out=None, forced_idx=None, scores_out=None, idx_out=None,
                    hidden_out=None, n_layers_run: int = 0, hidden_in=None, pos_in=None,
                    first_layer: int = 1, plan_L: int = 0, stream=None):
    opts = zsaa_forward_opts(_ptr(forced_idx), _ptr(scores_out), _ptr(idx_out), _ptr(hidden_out),
                             n_layers_run, _ptr(hidden_in), _ptr(pos_in), first_layer, plan_L)
    _check(lib().zsaa_forward_ex(model.handle, _ptr(token_ids), B, L, float(accel),
                                 _ptr(logits_out), _ptr(kept_pos_out), C.byref(opts),
                                 _stream(stream)))


def _lengths(lengths):
    arr = (C.c_int32 * len(lengths))(*[int(x) for x in lengths])
    return arr, len(lengths)


def zsaa_plan_varlen_config(cfg: zsaa_config, lengths, accel: float) -> Tuple[List[List[int]], float]:
    arr, B = _lengths(lengths)
    n1 = cfg.n_layers + 1
    sched = (C.c_int * (B * n1))()
    alpha = C.c_double()
    _check(lib().zsaa_plan_varlen_config(C.byref(cfg), C.cast(arr, C.c_void_p), B, float(accel), sched,
                                         C.byref(alpha)))
    return [list(sched[b * n1:(b + 1) * n1]) for b in range(B)], alpha.value


def zsaa_plan_varlen(model: Model, lengths, accel: float) -> Tuple[List[List[int]], float]:
    arr, B = _lengths(lengths)
    n1 = model.cfg.n_layers + 1
    sched = (C.c_int * (B * n1))()
    alpha = C.c_double()
    _check(lib().zsaa_plan_varlen(model.handle, C.cast(arr, C.c_void_p), B, float(accel), sched,
                                  C.byref(alpha)))
    return [list(sched[b * n1:(b + 1) * n1]) for b in range(B)], alpha.value


def zsaa_forward_varlen(model: Model, token_ids, lengths, accel: float, logits_out, kept_pos_out=None,
                        forced_idx=None, scores_out=None, idx_out=None, stream=None):
    """token_ids: device int32 [sum(lengths)] packed; lengths: host sequence of ints."""
    arr, B = _lengths(lengths)
    opts = None
    if forced_idx is not None or scores_out is not None or idx_out is not None:
        opts = C.byref(zsaa_forward_opts(_ptr(forced_idx), _ptr(scores_out), _ptr(idx_out), None,
                                         0, None, None, 0, 0))
    _check(lib().zsaa_forward_varlen(model.handle, _ptr(token_ids), C.cast(arr, C.c_void_p), B,
                                     float(accel), _ptr(logits_out), _ptr(kept_pos_out), opts,
                                     _stream(stream)))


def zsaa_forward_masked(model: Model, token_ids, B: int, L: int, accel: float, logits_out,
                        kept_pos_out=None, forced_pos=None, scores_out=None, idx_out=None,
                        stream=None):
    """Appendix B mode; forced_pos / idx_out hold kept POSITIONS per pruning layer."""
    opts = None
    if forced_pos is not None or scores_out is not None or idx_out is not None:
        opts = C.byref(zsaa_forward_opts(_ptr(forced_pos), _ptr(scores_out), _ptr(idx_out), None,
                                         0, None, None, 0, 0))
    _check(lib().zsaa_forward_masked(model.handle, _ptr(token_ids), B, L, float(accel),
                                     _ptr(logits_out), _ptr(kept_pos_out), opts, _stream(stream)))


def zsaa_forward_marked(model: Model, token_ids, B: int, L: int, accel: float, logits_out,
                        kept_pos_out=None, forced_pos=None, scores_out=None, idx_out=None,
                        stream=None):
    """Appendix B figure mode (marked rows may be reactivated); hooks as zsaa_forward_masked."""
    opts = None
    if forced_pos is not None or scores_out is not None or idx_out is not None:
        opts = C.byref(zsaa_forward_opts(_ptr(forced_pos), _ptr(scores_out), _ptr(idx_out), None,
                                         0, None, None, 0, 0))
    _check(lib().zsaa_forward_marked(model.handle, _ptr(token_ids), B, L, float(accel),
                                     _ptr(logits_out), _ptr(kept_pos_out), opts, _stream(stream)))


def zsaa_forward_host(model: Model, token_ids, B: int, L: int, accel: float, logits_out,
                      kept_pos_out=None, stream=None):
    """token_ids / logits_out / kept_pos_out are HOST buffers (numpy arrays or
    CPU tensors; pinned memory gives the fastest copies)."""

    def hp(a):
        if a is None:
            return None
        if hasattr(a, "data_ptr"):
            return a.data_ptr()
        return a.ctypes.data

    _check(lib().zsaa_forward_host(model.handle, hp(token_ids), B, L, float(accel), hp(logits_out),
                                   hp(kept_pos_out), _stream(stream)))


# ------------------------------------------------------------------ generation

class Cache:
    """Owns a zsaa_cache handle (pruned KV cache of one prompt batch)."""

    def __init__(self, model: Model, B: int, L: int, accel: float, max_new: int):
        h = C.c_void_p()
        _check(lib().zsaa_cache_create(model.handle, B, L, float(accel), max_new, C.byref(h)))
        self.handle = h
        self.model = model  # the cache must not outlive its model
        self.B, self.L, self.accel, self.max_new = B, L, accel, max_new

    def close(self):
        if getattr(self, "handle", None) is not None and self.handle.value:
            lib().zsaa_cache_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def zsaa_cache_create(model: Model, B: int, L: int, accel: float, max_new: int) -> Cache:
    return Cache(model, B, L, accel, max_new)


def zsaa_cache_destroy(cache: Cache):
    cache.close()


def zsaa_prefill(model: Model, cache: Cache, token_ids, logits_out, forced_idx=None,
                 scores_out=None, idx_out=None, stream=None):
    opts = None
    if forced_idx is not None or scores_out is not None or idx_out is not None:
        opts = C.byref(zsaa_forward_opts(_ptr(forced_idx), _ptr(scores_out), _ptr(idx_out), None,
                                         0, None, None, 0, 0))
    _check(lib().zsaa_prefill(model.handle, cache.handle, _ptr(token_ids), _ptr(logits_out), opts,
                              _stream(stream)))


def zsaa_decode_step(model: Model, cache: Cache, token_ids, logits_out, stream=None):
    _check(lib().zsaa_decode_step(model.handle, cache.handle, _ptr(token_ids), _ptr(logits_out),
                                  _stream(stream)))


def zsaa_cache_layer(cache: Cache, layer: int) -> Dict:
    """Device pointers (ints) k, v, pos and the sizes base, len, cap of one layer (1-based)."""
    k, v, pos = C.c_void_p(), C.c_void_p(), C.c_void_p()
    base, ln, cap = C.c_int(), C.c_int(), C.c_int()
    _check(lib().zsaa_cache_layer(cache.handle, layer, C.byref(k), C.byref(v), C.byref(pos),
                                  C.byref(base), C.byref(ln), C.byref(cap)))
    return dict(k=k.value, v=v.value, pos=pos.value, base=base.value, len=ln.value, cap=cap.value)


def zsaa_cache_bytes(cache: Cache) -> Tuple[int, int]:
    a, b = C.c_size_t(), C.c_size_t()
    _check(lib().zsaa_cache_bytes(cache.handle, C.byref(a), C.byref(b)))
    return a.value, b.value


def zsaa_trace_begin(model: Model):
    _check(lib().zsaa_trace_begin(model.handle))


def zsaa_trace_end(model: Model) -> List[Dict]:
    rows = (zsaa_trace_row * 64)()
    n = C.c_int()
    _check(lib().zsaa_trace_end(model.handle, rows, 64, C.byref(n)))
    return [dict(name=r.name.decode(), launches=r.launches, ms=r.ms, flops=r.flops, bytes=r.bytes)
            for r in rows[: min(n.value, 64)]]


def zsaa_sync(model: Model, stream=None):
    _check(lib().zsaa_sync(model.handle, _stream(stream)))


# ------------------------------------------------------------------ isolated ops

def zsaa_score_select(hidden, B: int, L: int, d: int, k: int, idx_out, gathered_out=None,
                      stream=None):
    _check(lib().zsaa_score_select(_ptr(hidden), B, L, d, k, _ptr(idx_out), _ptr(gathered_out),
                                   _stream(stream)))


def zsaa_score_select_ex(hidden, B: int, L: int, d: int, dtype: int, k: int, flags: int,
                         scores_in, scores_out, idx_out, gathered_out=None, stream=None):
    _check(lib().zsaa_score_select_ex(_ptr(hidden), B, L, d, dtype, k, flags, _ptr(scores_in),
                                      _ptr(scores_out), _ptr(idx_out), _ptr(gathered_out),
                                      _stream(stream)))


def zsaa_score_select_noalloc(hidden, B: int, L: int, d: int, k: int, idx_out, gathered_out=None,
                              stream=None):
    """zsaa_score_select without device allocation (fixed 4 MiB scratch, B*L <= 2**20)."""
    _check(lib().zsaa_score_select_noalloc(_ptr(hidden), B, L, d, k, _ptr(idx_out),
                                           _ptr(gathered_out), _stream(stream)))


def zsaa_op_linear(A, W, W2, resid, out, M: int, N: int, K: int, dtype: int, epilogue: int,
                   pos=None, rope_cols: int = 0, rope_hd: int = 0, rope_theta: float = 0.0,
                   stream=None):
    _check(lib().zsaa_op_linear(_ptr(A), _ptr(W), _ptr(W2), _ptr(resid), _ptr(out), M, N, K, dtype,
                                epilogue, _ptr(pos), rope_cols, rope_hd, float(rope_theta),
                                _stream(stream)))


def zsaa_gemm_schedule(epilogue: int, M: int, N: int, K: int, hd: int, sms: int, pair_slots: int,
                       split_slots: int):
    """Host-side tile plan of the tiled GEMM: (plan: 12 ints, items: list of
    8-int tuples (unit, tile, kb0, kb1, kind, slot, count, stride))."""
    plan = (C.c_int32 * 12)()
    n = C.c_int64()
    _check(lib().zsaa_gemm_schedule(epilogue, M, N, K, hd, sms, pair_slots, split_slots, plan, None, 0,
                                    C.byref(n)))
    buf = (C.c_int32 * (8 * max(n.value, 1)))()
    _check(lib().zsaa_gemm_schedule(epilogue, M, N, K, hd, sms, pair_slots, split_slots, plan, buf,
                                    n.value, C.byref(n)))
    flat = list(buf)
    return list(plan), [tuple(flat[8 * i:8 * i + 8]) for i in range(n.value)]


def zsaa_op_attention(qkv, B: int, N: int, Hq: int, Hkv: int, hd: int, dtype: int, out, lse,
                      stream=None):
    _check(lib().zsaa_op_attention(_ptr(qkv), B, N, Hq, Hkv, hd, dtype, _ptr(out), _ptr(lse),
                                   _stream(stream)))


def zsaa_op_colmass(qkv, lse, B: int, N: int, Hq: int, Hkv: int, hd: int, dtype: int, colmass,
                    stream=None):
    _check(lib().zsaa_op_colmass(_ptr(qkv), _ptr(lse), B, N, Hq, Hkv, hd, dtype, _ptr(colmass),
                                 _stream(stream)))


def zsaa_op_attention_ex(qkv, B: int, N: int, Hq: int, Hkv: int, hd: int, dtype: int, causal: bool,
                         out, lse, stream=None):
    _check(lib().zsaa_op_attention_ex(_ptr(qkv), B, N, Hq, Hkv, hd, dtype, 1 if causal else 0,
                                      _ptr(out), _ptr(lse), _stream(stream)))


def zsaa_op_colmass_ex(qkv, lse, B: int, N: int, Hq: int, Hkv: int, hd: int, dtype: int,
                       causal: bool, colmass, stream=None):
    _check(lib().zsaa_op_colmass_ex(_ptr(qkv), _ptr(lse), B, N, Hq, Hkv, hd, dtype,
                                    1 if causal else 0, _ptr(colmass), _stream(stream)))


def zsaa_device_status():
    _check(lib().zsaa_device_status())


def zsaa_selftest_wait_timeout(stream=None) -> int:
    """Run the bounded-wait self-test; returns its status code (ZSAA_ERR_TIMEOUT
    when a wait that nothing completes gives up and reports, as it should)."""
    return int(lib().zsaa_selftest_wait_timeout(_stream(stream)))


def zsaa_last_error() -> str:
    return lib().zsaa_last_error().decode()


def zsaa_version() -> str:
    return lib().zsaa_version().decode()
