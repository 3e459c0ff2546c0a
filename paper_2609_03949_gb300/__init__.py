"""GB300-native VestigeKV decode hot path: RoPE-branch scoring, per-head top-k selection and absorbed-MLA
sparse attention over a DeepSeek-style MLA cache, as hand-written sm_103a CUDA behind a C ABI (libvk.so).

``vk`` is the ctypes binding (same names as include/vk.h); ``datagen`` draws the seeded synthetic workloads.
Submodules are imported lazily so that the input generator can be used without the CUDA library.
"""
__all__ = ["vk", "datagen", "bytes_model"]
