"""GB300-native (sm_103a) implementation of JET's teacher-forced candidate-scoring step.

``jet`` is the ctypes binding of libjet (C ABI in ``include/jet.h``);
``step`` strings the entry points together into one scoring step.
"""
__all__ = ["jet", "step", "build"]
