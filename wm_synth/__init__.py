"""Seeded synthetic inputs shared by the oracle side and the GPU side.

Holds no arithmetic of the decode method: only workload shapes, a
counter-based value generator (host and device) and input builders.
"""
from . import configs, gen, inputs  # noqa: F401
