"""Seeded synthetic inputs for the tree-verification step.

Shared by the CUDA path's tests and benchmark and by the CPU checker; it draws
inputs only and holds none of the verification arithmetic.
"""

from . import configs, gen, model, trees  # noqa: F401
