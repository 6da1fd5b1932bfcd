"""qmla_mla_decode_static, the decode entry point that allocates nothing.

Some callers cannot allocate device memory at the point where they run the
decode: code inside an allocator-free region of a serving loop, or a host
library that is handed finished buffers and must not call cudaMalloc (it
synchronises and grows memory the caller does not control). For them the
library keeps the decode's scratch in one fixed device array. These tests call
it through the C ABI and check that it returns what qmla_mla_decode (which
takes a caller workspace) returns, within the same tolerance the parity tests
use, on two calls in a row with different queries.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2609_36760_gb300 as Q
from harness import TAU, Case, rel_l2
from workloads import synthetic as W

pytestmark = pytest.mark.gpu

MAX_ABS = 2e-3
REL_L2 = 1e-3


def _decode_static(case: Case, ql: torch.Tensor, qp: torch.Tensor, lens, out: torch.Tensor, lse: torch.Tensor,
                   batch: int | None = None) -> int:
    L = Q.lib()
    vp = ctypes.c_void_p
    sl = torch.tensor(lens, dtype=torch.int32, device="cuda")
    st = L.qmla_mla_decode_static(
        vp(case.pool.data_ptr()), case.w.c_bits, case.pool.shape[0], vp(ql.data_ptr()), vp(qp.data_ptr()),
        case.w.batch if batch is None else batch, case.w.heads, vp(case.table_d.data_ptr()),
        case.table_d.shape[1], vp(sl.data_ptr()), TAU, vp(out.data_ptr()), vp(lse.data_ptr()),
        vp(case.dev_err.data_ptr()), vp(torch.cuda.current_stream().cuda_stream))
    torch.cuda.synchronize()
    return st


def test_static_scratch_matches_workspace_entry_point():
    w = W.small_workload("noalloc", batch=6, heads=128, lengths=(4097, 300, 1, 2000, 64, 9000), seed=91)
    assert Q.decode_workspace_bytes(w.batch, w.heads) <= Q.static_scratch_bytes()
    c = Case(w)
    c.prefill_all()
    lens = c.lengths_at(0)
    for call in range(2):
        ql, qp = W.queries(w, call)
        ref_out, ref_lse = c.decode(0, queries=(ql, qp))  # workspace entry point
        ql_d, qp_d = ql.contiguous().cuda(), qp.contiguous().cuda()
        out = torch.full((w.batch, w.heads, 512), float("nan"), dtype=torch.float32, device="cuda")
        lse = torch.full((w.batch, w.heads), float("nan"), dtype=torch.float32, device="cuda")
        assert _decode_static(c, ql_d, qp_d, lens, out, lse) == 0
        got, got_lse = out.cpu().numpy(), lse.cpu().numpy()
        assert np.isfinite(got).all()
        assert np.max(np.abs(got - ref_out)) <= MAX_ABS
        assert rel_l2(got, ref_out) <= REL_L2
        assert np.max(np.abs(got_lse - ref_lse)) <= 1e-3
    assert c.dev_error() == 0


def test_static_scratch_rejects_oversized_requests():
    w = W.small_workload("noalloc2", batch=2, heads=16, lengths=(64, 64), seed=92)
    c = Case(w)
    c.prefill_all()
    ql, qp = W.queries(w, 0)
    out = torch.zeros((w.batch, w.heads, 512), dtype=torch.float32, device="cuda")
    lse = torch.zeros((w.batch, w.heads), dtype=torch.float32, device="cuda")
    before = out.clone()
    # A batch whose scratch cannot fit is refused before anything is launched.
    st = _decode_static(c, ql.contiguous().cuda(), qp.contiguous().cuda(), [64, 64], out, lse, batch=1 << 20)
    assert st == 3  # QMLA_ERR_WORKSPACE_TOO_SMALL
    assert torch.equal(out, before)
