"""GB300 FASGD parameter server: C-ABI CUDA library + thin Python binding.

``paper_1601_04033_gb300.fasgd`` is the ctypes binding of include/fasgd.h
(import it after building the library); ``streams`` draws the seeded
synthetic workloads; ``build`` compiles the library with nvcc for sm_103a.
"""
