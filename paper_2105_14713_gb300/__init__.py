"""GB300-native forward convolution of 1xN-pruned layers (Lin et al., 1xN pruning).

``onexn``   -- ctypes binding of the C ABI in include/onexn.h (libonexn.so)
``layer``   -- PrunedConv2d: prune + pack on the host, conv on the GPU
``workloads`` -- seeded synthetic layer shapes and inputs
"""
__all__ = ["onexn", "layer", "workloads"]
