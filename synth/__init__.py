"""Seeded synthetic inputs shaped like the paper's workloads (no method arithmetic)."""
from .configs import (ALL, STACK4_7800, TINY_256, WAN_BLOCK_32760, WAN_STACK40_32760,
                      WAN_SWEEP_63960, Workload, small)
from . import generate

__all__ = ["ALL", "STACK4_7800", "TINY_256", "WAN_BLOCK_32760", "WAN_STACK40_32760",
           "WAN_SWEEP_63960", "Workload", "small", "generate"]
