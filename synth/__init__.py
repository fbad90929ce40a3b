"""Seeded synthetic inputs for the verification step (shared by tests, the oracle
side and the CUDA side; holds none of the step's arithmetic)."""

from . import rng, trees, workloads  # noqa: F401
