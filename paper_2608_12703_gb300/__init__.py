"""GB300 (sm_103a) draft-verify step for single-model speculative ASR decoding.

``asrspec``: ctypes binding of the C ABI (include/asrspec.h).
``session``: a small driver that owns device buffers and runs decode loops.
``build``:   compiles libasrspec.so in-tree with nvcc.
"""
