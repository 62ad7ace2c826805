"""GB300-native (sm_103a) ALR slot-loss hot path: CUDA kernels behind a C ABI (libalr)
and a thin ctypes binding (``paper_2609_38795_gb300.alr``)."""
