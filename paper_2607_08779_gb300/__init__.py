"""GB300-native signed symmetric few-bit weight path.

Group-wise q-bit (q = 2/3/4) weight quantization with the signed absmax
sign rule, and the decode GEMV / prefill GEMM that consume the packed codes,
as hand-written sm_103a CUDA kernels behind the C ABI in include/sss.h.
Submodules: ``sss`` (the ctypes binding; it loads libsss.so on first use) and
``inputs`` (seeded synthetic inputs).
"""
