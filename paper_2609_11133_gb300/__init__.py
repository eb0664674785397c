"""GB300-native MoE decode layer: hand-written sm_103a CUDA behind a C ABI.

The CUDA library (``_build/libmoe.so``) is built by ``build.build()`` and
bound by ``binding``.  ``synth`` makes seeded synthetic inputs.
"""
