"""Seeded synthetic inputs for MLKV decode: the one module that feeds both the oracle and the CUDA
library.  It holds no attention arithmetic; see ``gen`` for the generator's definition."""
from . import gen, workloads  # noqa: F401
