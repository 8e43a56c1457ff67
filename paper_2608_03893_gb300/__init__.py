"""kvx: GB300-native cross-model KV-cache mapper (arXiv 2608.03893).

The mapper turns a source model's prefilled KV cache into a same-family target
model's KV cache (Sec. 3: top-k source layers per target layer, RoPE strip, per-head
ridge map X W + b, target RoPE).  The compute runs in hand-written CUDA for sm_103a
behind the C ABI declared in ``include/kvx.h``; ``paper_2608_03893_gb300.kvx`` is the
thin ctypes binding.  Importing this package loads nothing; the binding loads the
shared library on first use and raises if it is missing.
"""
