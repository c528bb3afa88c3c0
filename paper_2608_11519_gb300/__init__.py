"""GB300-native FLARE++ routing chain (libflarepp) and its Python binding.

Importing the package loads nothing native; ``paper_2608_11519_gb300.flarepp`` loads the
CUDA library on first use and raises if it is missing.
"""
