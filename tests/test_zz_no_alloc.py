"""The allocation-free entry point, opattn_prefill_noalloc.

Some callers cannot let a library allocate device memory: an engine that has
reserved nearly all of HBM for its KV cache and serves every allocation from
its own pool, or a process held to a device-memory quota.  For them the
library keeps the work list in a fixed device array instead of per-call
scratch.  These tests check that entry point against opattn_prefill.  The
file is named so that pytest collects it last.
"""
import numpy as np
import pytest
import torch

import paper_2608_13499_gb300 as pkg
from paper_2608_13499_gb300 import build as pbuild
from paper_2608_13499_gb300 import workloads as W

O_MAX, O_MEAN, LSE_MAX = 1e-2, 1e-3, 1e-3


@pytest.fixture(scope="module", autouse=True)
def lib():
    pbuild.build()
    return pkg.load()


def _outputs(w, dev):
    o = torch.full((w.total_q, w.Hq, w.d), float("nan"), dtype=torch.bfloat16, device=dev)
    lse = torch.full((w.total_q, w.Hq), float("nan"), dtype=torch.float32, device=dev)
    return o, lse


def _close(o_a, l_a, o_b, l_b):
    oa, ob = o_a.float().cpu().numpy(), o_b.float().cpu().numpy()
    assert np.all(np.isfinite(oa))
    err = np.abs(oa - ob)
    assert err.max() <= O_MAX and err.mean() <= O_MEAN
    la, lb = l_a.cpu().numpy(), l_b.cpu().numpy()
    fin = np.isfinite(lb)
    assert np.array_equal(np.isfinite(la), fin)
    assert np.all(la[~fin] == -np.inf)
    if fin.any():
        assert np.abs(la[fin] - lb[fin]).max() <= LSE_MAX
    # the same kernel runs the same work list, so every row comes out bit for bit the same
    assert torch.equal(o_a, o_b) and torch.equal(l_a, l_b)


@pytest.mark.gpu
def test_noalloc_matches_opattn_prefill_on_two_calls_in_a_row():
    # a larger batch first, then a smaller one, so that the second call
    # runs over what the first left in the shared array
    work = [W.llama3_8b(), W.Workload("noalloc_small", [1, 130, 77, 0, 300], [1, 130, 200, 5, 300], 16, 4, 128)]
    inputs, ref, got = [], [], []
    for w in work:
        q, k, v = W.make_inputs(w, "cuda")
        inputs.append((q, k, v))
        o, lse = _outputs(w, "cuda")
        pkg.opattn_prefill(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
        ref.append((o, lse))
    torch.cuda.synchronize()
    for w, (q, k, v) in zip(work, inputs):  # two calls in a row on one stream
        o, lse = _outputs(w, "cuda")
        pkg.opattn_prefill_noalloc(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
        got.append((o, lse))
    torch.cuda.synchronize()
    for (o_r, l_r), (o_g, l_g) in zip(ref, got):
        _close(o_g, l_g, o_r, l_r)


def test_noalloc_rejects_batches_beyond_its_capacity_before_touching_the_gpu():
    # G = 1 gives 256 tokens per unit: 64 kv heads x 513 blocks > 32768 units.
    # The pointers are never dereferenced: the size check comes first.
    A = 0x10000
    n_tok = 513 * 256
    st = pkg.opattn_prefill_noalloc(A, A, A, A, A, [0, n_tok], [0, n_tok], 1, 64, 64, 128, 0.088,
                                    stream=0, check=False)
    assert st == pkg.OPATTN_ERR_CAPACITY
