"""GB300-native server-side hot path of FedOptima (arxiv 2504.13850).

The compute path lives in the C-ABI shared library built from ``csrc/``;
``api`` is a thin ctypes binding over it.
"""
