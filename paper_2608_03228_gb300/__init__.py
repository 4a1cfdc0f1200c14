"""GB300-native SAKI score-map retrieval: C-ABI CUDA library plus a thin binding.

Import ``paper_2608_03228_gb300.saki`` for the binding (it loads the CUDA
library); ``paper_2608_03228_gb300.synth`` holds the seeded input generators.
"""
