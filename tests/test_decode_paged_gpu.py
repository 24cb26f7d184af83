"""GPU parity of decode over paged K/V caches (opattn_decode_paged) against the fp64 oracle.

The caches are built from the packed K/V the oracle reads: every sequence's
pages are scattered in a seeded random order over a pool with spare pages,
and every row no sequence owns holds a constant, so a page read from the
wrong place changes the result.  Cases cover page sizes 8 to 128, key
counts that end inside a page, several query tokens, split key ranges, a
plan run repeatedly, and the full-size paged workload on sampled rows.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_13499_gb300 as pkg
from paper_2608_13499_gb300 import workloads as W

pytestmark = pytest.mark.gpu

O_MAX, O_MEAN, LSE_MAX = 1e-2, 1e-3, 1e-3


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_13499_gb300 import build as pbuild
    pbuild.build()
    pkg.load()
    oracle.build()


def check(o_gpu, lse_gpu, o_ref, lse_ref, what=""):
    o = o_gpu.float().cpu().numpy().astype(np.float64)
    lse = lse_gpu.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(o)), f"{what}: non-finite O"
    err = np.abs(o - o_ref)
    assert err.max() <= O_MAX, f"{what}: O max-abs {err.max():.3e}"
    assert err.mean() <= O_MEAN, f"{what}: O mean-abs {err.mean():.3e}"
    fin = np.isfinite(lse_ref)
    assert np.array_equal(np.isfinite(lse), fin), f"{what}: LSE finiteness differs"
    if fin.any():
        lerr = np.abs(lse[fin] - lse_ref[fin]).max()
        assert lerr <= LSE_MAX, f"{what}: LSE max-abs {lerr:.3e}"


def paged_inputs(w, page, seed=0):
    q, k, v = W.make_inputs(w, "cuda")
    lay = W.paged_layout(w.k_lens, page, seed=seed)
    kc, vc = W.to_paged(k, w.k_lens, lay), W.to_paged(v, w.k_lens, lay)
    table = torch.from_numpy(lay.block_table).to("cuda")
    return q, k, v, kc, vc, table, lay


def run_paged(w, q, kc, vc, table, lay):
    o = torch.full((w.total_q, w.Hq, w.d), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((w.total_q, w.Hq), float("nan"), dtype=torch.float32, device="cuda")
    pkg.opattn_decode_paged(q, kc, vc, table, lay.num_blocks, lay.page_size, lay.max_blocks, o, lse, w.cu_q,
                            np.asarray(w.k_lens, dtype=np.int32), w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    torch.cuda.synchronize()
    return o, lse


CASES = [
    (8, [1] * 5, [7, 8, 9, 1000, 3001]),
    (16, [1] * 6, [1, 15, 16, 17, 4100, 700]),
    (64, [2, 2, 2], [63, 2000, 129]),
    (128, [4, 1, 1], [5000, 127, 128]),
    (16, [1, 3], [40000, 12000]),               # long: split into chunks and merged
]


@pytest.mark.parametrize("case", CASES, ids=[f"page{c[0]}_{len(c[1])}seq" for c in CASES])
def test_paged_matches_oracle(case):
    page, lq, lk = case
    w = W.Workload(f"paged{page}", lq, lk, 16, 2, 128, 1.0, page)
    q, k, v, kc, vc, table, lay = paged_inputs(w, page, seed=page)
    o, lse = run_paged(w, q, kc, vc, table, lay)
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    check(o, lse, o_ref, lse_ref, w.name)


def test_paged_equals_packed_decode():
    """Same keys in a packed tensor and in a shuffled paged cache: the two results agree."""
    w = W.Workload("paged_vs_packed", [1, 2, 1], [3000, 517, 64], 32, 8, 128, 1.0, 4)
    q, k, v, kc, vc, table, lay = paged_inputs(w, 32, seed=9)
    o_p, lse_p = run_paged(w, q, kc, vc, table, lay)
    o_d = torch.empty_like(o_p)
    lse_d = torch.empty_like(lse_p)
    pkg.opattn_decode(q, k, v, o_d, lse_d, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    torch.cuda.synchronize()
    assert (o_p.float() - o_d.float()).abs().max().item() <= 1e-2
    assert (lse_p - lse_d).abs().max().item() <= 1e-3


def test_paged_plan_runs_repeatedly_and_rejects_packed_runs():
    w = W.Workload("paged_plan", [1, 1], [20000, 333], 16, 2, 128, 1.0, 5)
    q, k, v, kc, vc, table, lay = paged_inputs(w, 16, seed=5)
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    o = torch.empty((w.total_q, w.Hq, w.d), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((w.total_q, w.Hq), dtype=torch.float32, device="cuda")
    with pkg.Plan(w.cu_q, np.asarray(w.k_lens, dtype=np.int32), w.Hq, w.Hkv, w.d, decode=True, block_size=16,
                  max_blocks=lay.max_blocks) as plan:
        assert plan.paged and plan.n_units > 2
        with pytest.raises(pkg.OpattnError):
            plan.run(q, k, v, o, lse, w.scale)            # a paged plan needs the block table
        for _ in range(3):
            o.fill_(float("nan"))
            plan.run_paged(q, kc, vc, table, lay.num_blocks, o, lse, w.scale)
        torch.cuda.synchronize()
    check(o, lse, o_ref, lse_ref, "paged plan x3")
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=True) as packed:
        with pytest.raises(pkg.OpattnError):
            packed.run_paged(q, kc, vc, table, lay.num_blocks, o, lse, w.scale)


def test_full_size_paged_workload_on_sampled_rows():
    w = W.decode_llama3_70b_paged16()
    q, k, v, kc, vc, table, lay = paged_inputs(w, w.page_size, seed=w.seed)
    o, lse = run_paged(w, q, kc, vc, table, lay)
    assert torch.isfinite(o.float()).all().item()
    rng = np.random.default_rng(1)
    tok = rng.integers(0, w.total_q, 40)
    hd = rng.integers(0, w.Hq, 40)
    o_r, lse_r = oracle.attention_rows(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale,
                                       tok, hd)
    check(o[tok, hd], lse[tok, hd], o_r, lse_r, w.name)
