"""CPU oracle for the branch-cached MoE layer (MoECa).

TEST INFRASTRUCTURE.  Only the tests, the package smoke check and the CPU
baseline leg of the benchmark may import anything here; the product path (the
CUDA library and its Python binding) never does, and shares no code with it.
"""
