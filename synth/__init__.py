"""Seeded synthetic inputs shared by the tests, the benchmark and the oracle checks.

This package draws random logits, masks and nothing else: it holds none of the
loss, acceptance or reward arithmetic, so both the CUDA path and the CPU oracle
can consume the very same bytes without sharing any of the method's code.
"""

from .workloads import (  # noqa: F401
    REWARD,
    SEQUENCES,
    SeqWorkload,
    WORKLOADS,
    Workload,
    bytes_per_tensor,
    make_logits,
    make_reward_logits,
    make_seq_logits,
    workload,
)
