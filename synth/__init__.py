"""Seeded synthetic inputs shared by the oracle tests and the CUDA path."""
from . import gen, workloads  # noqa: F401
