"""Seeded synthetic inputs (shapes, weights, latents, trajectories, stand-in
response tables).  Holds none of the method's arithmetic; both the oracle and
the CUDA path's tests and benchmark draw their inputs from here."""

from .configs import WORKLOADS, Workload  # noqa: F401
from . import gen  # noqa: F401
