"""Seeded synthetic inputs for the low-bit MLA decode path.

This package only draws random numbers and lays out block tables; it holds none
of the method's arithmetic (no quantisation, packing, dequantisation or
attention). Both the CPU oracle (through the tests) and the CUDA library consume
the exact bf16 tensors produced here.
"""
from .synthetic import (  # noqa: F401
    WORKLOADS,
    Workload,
    block_table,
    channel_gains,
    kpe_for_seq,
    latent_for_seq,
    queries,
    seq_lengths,
    small_workload,
)
