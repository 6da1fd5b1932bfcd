"""CPU oracle for the low-bit MLA decode path (test infrastructure).

This package is the independent, slow, obviously-correct definition that the
CUDA library is checked against. It is test infrastructure: only ``tests/``,
``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
or run it. The product path never calls it, and it shares no code, constants
or helpers with ``paper_2609_36760_gb300``.

Modules
-------
quantizer  per-token group-64 asymmetric quantiser and bit packing (App. C.4)
layout     this library's 64-token block byte layout, writer and reader
attention  dequantisation, absorbed MLA decode attention in fp64 (Eq. mla_compact)
           and the split-result merge (App. C.5, global attention normalisation)
storage    the persistent-storage closed form (App. C.5, Eq. physical_cache_storage)
protection sink4/local128 BF16 protection: the protected set, this library's
           protection-buffer rows and writer rule, protected attention (App. C.5,
           "BF16 protection and cache lifecycle")
paper_format the paper's own 20,480-byte page: bf16 content scales, fp32 RoPE
           scale, uint8 zero points, its quantiser staging, writer and reader
           (App. C.4, App. C.5 storage layout)
multi_query decode with T query tokens per sequence: Eq. mla_compact with its
           additive causal mask, masked partials and their merge (App. C.5)
fusion     offline-fusion identities: content rotation/scale with compensated
           consumers (Eq. content_transform, App. C.1), Prop. 1's reciprocal
           RoPE-pair transform and its commutation with RoPE (App. C.2)

Every function is pinned by tests under ``tests/test_oracle_*.py``; nothing in
this package is marked "parity unpinned".
"""
from . import attention, fusion, layout, multi_query, paper_format, protection, quantizer, storage  # noqa: F401
