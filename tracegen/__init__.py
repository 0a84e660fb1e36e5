"""Seeded synthetic inputs for the DualMap routing path (shared by the CUDA
path's tests/bench and by the CPU oracle's tests; holds none of the method)."""
from .configs import WORKLOADS, ORDER, workload
from .trace import Trace, piece_tokens, mix64, ALIGN_TOKENS
