"""GB300-native branch-cached DiT-MoE layer stack (MoECa).

``moeca`` binds the CUDA library (libmoeca.so, C ABI in include/moeca.h),
``workloads`` makes seeded synthetic inputs and ``build`` compiles the library.
Import ``paper_2606_15615_gb300.moeca`` explicitly: it loads the library and
fails loudly if it has not been built.
"""
