"""GB300-native SkewAdam: tiered optimizer state for MoE training (libskewadam).

``skewadam`` is the ctypes binding of the C ABI in ``include/skewadam.h``;
``workloads`` draws the seeded synthetic parameter sets.
"""
