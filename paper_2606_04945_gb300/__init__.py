"""GB300 (sm_103a) hot path of STaR-Quant: the SGAT W4A4 linear and TAC.

The computation lives in libstarq.so (CUDA kernels behind the C ABI declared
in include/starq.h). ``paper_2606_04945_gb300.abi`` is its Python binding,
``paper_2606_04945_gb300.inputs`` the seeded synthetic workloads, and
``paper_2606_04945_gb300.build`` the in-tree nvcc build. Importing the
package itself loads nothing.
"""
