"""GB300-native diffusion-LM lossless compression (sm_103a CUDA + C ABI).

``paper_2608_11249_gb300.dlmz`` is the Python binding of the C-ABI library
``libdlmz.so`` (built by ``paper_2608_11249_gb300.build``); importing it
fails loudly when the library is missing.  ``sources`` holds the seeded
synthetic inputs.
"""
