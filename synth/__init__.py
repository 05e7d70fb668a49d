"""Seeded synthetic inputs shared by the oracle tests, the CUDA path tests and the bench."""
from .workloads import CONFIGS, Workload, sweep2048, rng  # noqa: F401
