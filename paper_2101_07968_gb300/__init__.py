"""GB300-native batched DynaComm scheduler (Cai et al., arXiv 2101.07968).

Exact forward (Eq. 8, Algorithm 3) and backward (Eq. 9, Algorithm 4) dynamic
programs for very many independent layer-wise communication scheduling
instances, a seeded profile generator and the timeline cost function f_m, all
as sm_103a CUDA kernels behind the C ABI of include/dynacomm.h.

``paper_2101_07968_gb300.dynacomm`` is the binding (loads libdynacomm.so);
``paper_2101_07968_gb300.workloads`` describes synthetic inputs only and loads
no native code.
"""
__all__ = ["dynacomm", "workloads", "build"]
