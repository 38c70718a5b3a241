"""GB300-native HiLo-Token hot path: frequency score, keep/pool split, pack,
compressed MMDiT block and unpack, as sm_103a CUDA behind a C ABI.

Importing the package does not load the CUDA library; ``hilo`` does.
"""
