"""Seeded synthetic-input generator shared by the CUDA path's tests/bench and the oracle."""
from .synth import *  # noqa: F401,F403
from .synth import WORKLOADS, Workload, get_workload, shrink, sweep_workload  # noqa: F401
