"""GPU parity of the prefill kernel over paged K/V caches (opattn_prefill_paged).

The typical use is chunked prefill in a paged serving engine: a chunk of a
prompt attends to its prefix, which already sits in the paged cache.  Caches
are built from the packed K/V the oracle reads, with every sequence's pages
scattered in a seeded random order and a constant in every row no sequence
owns.  Besides the oracle, the paged result must equal the packed-layout
result bit for bit: the kernel sees the same key rows in the same order.
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
        assert np.abs(lse[fin] - lse_ref[fin]).max() <= LSE_MAX, what


def run_both(w, page, seed):
    q, k, v = W.make_inputs(w, "cuda")
    lay = W.paged_layout(w.k_lens, page, seed=seed)
    kc, vc = W.to_paged(k, w.k_lens, lay), W.to_paged(v, w.k_lens, lay)
    table = torch.from_numpy(lay.block_table).to("cuda")
    o_p = torch.full((w.total_q, w.Hq, w.d), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse_p = torch.full((w.total_q, w.Hq), float("nan"), dtype=torch.float32, device="cuda")
    pkg.opattn_prefill_paged(q, kc, vc, table, lay.num_blocks, page, lay.max_blocks, o_p, lse_p, w.cu_q,
                             np.asarray(w.k_lens, dtype=np.int32), w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    o_d = torch.empty_like(o_p)
    lse_d = torch.empty_like(lse_p)
    pkg.opattn_prefill(q, k, v, o_d, lse_d, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    torch.cuda.synchronize()
    return (q, k, v), (o_p, lse_p), (o_d, lse_d), (kc, vc, table, lay)


CASES = [
    # (page, q_lens, k_lens, Hq, Hkv, d)
    (16, [512, 100, 1, 37], [812, 228, 1001, 37], 16, 2, 128),   # chunks over cached prefixes
    (64, [300, 64], [300, 700], 32, 8, 128),
    (128, [129, 255], [1000, 255], 16, 4, 128),
    (8, [70, 3, 200], [70, 90, 1300], 8, 8, 64),
    (32, [9, 0, 40, 5], [3, 0, 40, 0], 12, 4, 128),              # Lq > Lk, empty sequences, G = 3
]


@pytest.mark.parametrize("case", CASES, ids=[f"page{c[0]}_d{c[5]}_{len(c[1])}seq" for c in CASES])
def test_paged_prefill_matches_oracle_and_packed_bits(case):
    page, lq, lk, Hq, Hkv, d = case
    w = W.Workload(f"pp{page}", lq, lk, Hq, Hkv, d, 1.0, page)
    (q, k, v), (o_p, lse_p), (o_d, lse_d), _ = run_both(w, page, seed=page + 1)
    assert torch.equal(o_p.view(torch.int16), o_d.view(torch.int16))
    assert torch.equal(lse_p.view(torch.int32), lse_d.view(torch.int32))
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    check(o_p, lse_p, o_ref, lse_ref, w.name)


def test_paged_prefill_plan():
    w = W.Workload("pp_plan", [512, 200], [4000, 200], 16, 2, 128, 1.0, 31)
    (q, k, v), _, (o_d, lse_d), (kc, vc, table, lay) = run_both(w, 16, seed=31)
    o = torch.empty_like(o_d)
    lse = torch.empty_like(lse_d)
    with pkg.Plan(w.cu_q, np.asarray(w.k_lens, dtype=np.int32), w.Hq, w.Hkv, w.d, block_size=16,
                  max_blocks=lay.max_blocks) as plan:
        assert plan.paged and not plan.decode
        with pytest.raises(pkg.OpattnError):
            plan.run(q, k, v, o, lse, w.scale)
        for _ in range(2):
            o.fill_(float("nan"))
            plan.run_paged(q, kc, vc, table, lay.num_blocks, o, lse, w.scale)
        torch.cuda.synchronize()
    assert torch.equal(o.view(torch.int16), o_d.view(torch.int16))
    assert torch.equal(lse.view(torch.int32), lse_d.view(torch.int32))


def test_full_size_chunked_workload_paged():
    w = W.chunked()
    (q, k, v), (o_p, lse_p), (o_d, lse_d), _ = run_both(w, 16, seed=5)
    assert torch.equal(o_p.view(torch.int16), o_d.view(torch.int16))
    assert torch.equal(lse_p.view(torch.int32), lse_d.view(torch.int32))
    rng = np.random.default_rng(2)
    tok = rng.integers(0, w.total_q, 40)
    hd = rng.integers(0, w.Hq, 40)
    o_r, lse_r = oracle.attention_rows(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale,
                                       tok, hd)
    check(o_p[tok, hd], lse_p[tok, hd], o_r, lse_r, w.name)
