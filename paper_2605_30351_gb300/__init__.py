"""VideoMLA latent KV cache and absorbed-form MLA attention on GB300 (sm_103a).

The compute lives in ``libvideomla.so`` (CUDA kernels behind a C ABI, see
``include/videomla.h``); ``videomla`` is its ctypes binding and ``synth``
draws seeded synthetic workloads.
"""
