"""GB300-native pruned prefill (Zero-Shot Adjustable Acceleration, arXiv 2509.01190).

``zsaa`` is the ctypes binding of the C-ABI library ``lib/libzsaa.so`` (built
from ``csrc/`` by ``build.py``); ``inputs`` draws the seeded synthetic inputs.
Importing the package does not load the library; ``zsaa.lib()`` does.
"""
