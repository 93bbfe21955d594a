"""GB300-native Draft-Guided Eviction: the score -> select -> compact pass.

The computation lives in libdge.so (hand-written sm_103a CUDA kernels behind
the C ABI of include/dge.h); this package holds its build script, a ctypes
binding with the same call names, a small PyTorch-facing API, and the seeded
synthetic input generator.
"""
from .api import (Problem, compact, device_status, evict, problem_from_workload,  # noqa: F401
                  pyramid_budgets, score, select, workspace)
from .binding import DgeError  # noqa: F401
