"""Failure path without a GPU fault: a test-only flag makes one kernel wait on
a barrier that nothing arrives on.  The wait gives up after ~20 ms, the kernel
records a timeout in its status word, lets its copies in flight land, frees
TMEM and returns; the host reports OPATTN_ERR_TIMEOUT and the context stays
usable for the next call."""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_13499_gb300 as pkg
from paper_2608_13499_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_13499_gb300 import build as pbuild
    pbuild.build()
    oracle.build()


def test_forced_wait_timeout_is_reported_and_context_survives():
    w = W.Workload("fault", [200, 64], [200, 64], 8, 2, 128)
    q, k, v = W.make_inputs(w, "cuda")
    o = torch.zeros((w.total_q, w.Hq, w.d), dtype=torch.bfloat16, device="cuda")
    lse = torch.zeros((w.total_q, w.Hq), dtype=torch.float32, device="cuda")
    st = pkg.opattn_prefill_checked(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale,
                                    flags=pkg.OPATTN_FLAG_TEST_FORCE_TIMEOUT)
    assert st == pkg.OPATTN_ERR_TIMEOUT
    # the same context computes correctly afterwards, and the checked path reports OK
    st = pkg.opattn_prefill_checked(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    assert st == pkg.OPATTN_OK
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    err = np.abs(o.float().cpu().numpy() - o_ref)
    assert err.max() <= 1e-2 and err.mean() <= 1e-3
    assert np.abs(lse.cpu().numpy() - lse_ref).max() <= 1e-3
