"""libqvla: the Omega-QVLA W4A4 quantized linear (online Hadamard rotation, symmetric int4
activation quantisation with per-token or per-step scales, int4 x int4 GEMM, dequantisation)
as hand-written CUDA for GB300 (sm_103a) behind a C ABI (include/qvla.h).

``paper_2605_28803_gb300.qvla`` is the ctypes binding; ``workloads`` draws the synthetic
inputs; ``build`` compiles the library in-tree.
"""
