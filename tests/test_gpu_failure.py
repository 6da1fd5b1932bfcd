"""Failure detection without a GPU fault: a bounded pipeline wait that runs out
(a barrier phase nothing completes) reports QMLA_DEVERR_TIMEOUT and its site bit
in the caller's error word and returns, and the context stays usable; the
decode after it is correct."""
import time

import numpy as np
import pytest
import torch

import paper_2609_36760_gb300 as Q
from harness import Case, rel_l2
from workloads import synthetic as W

pytestmark = pytest.mark.gpu


def test_wait_runs_out_and_the_context_survives():
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    t0 = time.perf_counter()
    Q.debug_wait_timeout(2000, err)  # 2 ms
    torch.cuda.synchronize()
    assert time.perf_counter() - t0 < 5.0
    e = Q.read_dev_err(err)
    assert e & Q.DEVERR_TIMEOUT and e & Q.DEVERR_SITE_SOFTMAX, hex(e)
    # the same context decodes correctly afterwards
    c = Case(W.WORKLOADS["tiny_b1_h16_l256_int4"])
    c.prefill_all()
    out, lse = c.decode(0, lens=c.prefill)
    assert c.dev_error() == 0
    ref, rlse = c.oracle_decode(0, c.prefill[0])
    assert np.max(np.abs(out[0] - ref)) <= 2e-3 and rel_l2(out[0], ref) <= 1e-3
