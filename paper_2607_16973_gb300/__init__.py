"""GB300-native TurboQuant search path (rotate, quantise, pack; filtered top-k scan).

The compute runs in the CUDA library `libtq.so` built from `csrc/`; this package
is a thin binding over its C ABI (see include/tq.h).
"""
