"""GB300-native Free Energy Mixer forward read (arXiv 2602.07160).

The read o_{t,j} = (1/beta_j)(LSE_i(s_{t,i} + beta_j v_{i,j}) - LSE_i s_{t,i})
with the softmax prior s = QK^T/sqrt(d) runs in hand-written sm_103a CUDA
kernels behind a C ABI (``include/fem.h``, ``libfem.so``).  ``fem`` holds the
thin Python binding; importing this package does not load the library.
"""
__all__ = ["fem", "workloads"]
