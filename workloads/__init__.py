"""Seeded synthetic inputs shaped like the paper's MLLM revisit workloads.

Used by the tests, the benchmark and the oracle's checks alike; it creates
inputs only and computes no part of the method.
"""
from .configs import ALL, Workload, get  # noqa: F401
from .gen import CANARY_BITS, Batch, make_batch, make_decode_inputs, token_coords  # noqa: F401
