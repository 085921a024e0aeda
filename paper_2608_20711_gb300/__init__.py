"""GB300-native differential-oracle hot path (AsmEvo, arXiv 2608.20711):
Tier 1 guarded input synthesis and the per-element equivalence check of
Eq. 1, as CUDA kernels for sm_103a behind the C ABI of include/asmv.h.

`asmv` is the ctypes binding, `build` compiles libasmv.so in-tree and
`workloads` holds the seeded synthetic workload generators."""
