"""Seeded random batches against the fp64 oracle (GPU), every element.

Shapes are drawn from a fixed-seed generator: head dims 64 and 128, group
sizes G = Hq / Hkv that tile a 32-row warp evenly (1, 2, 4, ..., 128) and
ones that do not (3, 5, 6, 12), ragged lengths with empty sequences, cached
prefixes (Lk > Lq) and rows that see no key (Lq > Lk).  Prefill-shaped
batches go through opattn_prefill; decode-shaped ones (G * Lq <= 32) through
both opattn_prefill and opattn_decode, which must agree with the oracle
alike.  Same bar as the other parity tests.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_13499_gb300 as pkg
from paper_2608_13499_gb300 import workloads as W

pytestmark = pytest.mark.gpu

O_MAX, O_MEAN, LSE_MAX = 1e-2, 1e-3, 1e-3
GROUPS = [1, 2, 3, 4, 5, 6, 8, 12, 16, 32, 64, 128]


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2608_13499_gb300 import build as pbuild
    pbuild.build()
    pkg.load()
    oracle.build()


def prefill_case(i):
    rng = np.random.default_rng(1000 + i)
    d = int(rng.choice([64, 128]))
    G = int(rng.choice(GROUPS))
    Hkv = int(rng.choice([h for h in (1, 2, 4, 8) if G * h <= 128]))
    n_seq = int(rng.integers(1, 6))
    lq, lk = [], []
    for _ in range(n_seq):
        kind = rng.random()
        L = int(rng.integers(0, 300))
        if kind < 0.15:
            lq.append(L), lk.append(L // 3)                         # Lq > Lk: early rows see no key
        elif kind < 0.55:
            lq.append(L), lk.append(L + int(rng.integers(0, 400)))  # cached prefix
        else:
            lq.append(L), lk.append(L)
    return W.Workload(f"rand_prefill_{i}", lq, lk, G * Hkv, Hkv, d, 1.0, 2000 + i)


def decode_case(i):
    rng = np.random.default_rng(3000 + i)
    G = int(rng.choice([1, 2, 4, 8, 16, 32]))
    Hkv = int(rng.choice([h for h in (1, 2, 4, 8) if G * h <= 128]))
    n_seq = int(rng.integers(1, 9))
    max_q = 32 // G
    lq = [int(rng.integers(0, max_q + 1)) for _ in range(n_seq)]
    lk = [int(rng.integers(0, 3000)) if rng.random() < 0.9 else 0 for _ in range(n_seq)]
    return W.Workload(f"rand_decode_{i}", lq, lk, G * Hkv, Hkv, 128, 1.0, 4000 + i)


def outputs(w, device):
    o = torch.full((w.total_q, w.Hq, w.d), float("nan"), dtype=torch.bfloat16, device=device)
    lse = torch.full((w.total_q, w.Hq), float("nan"), dtype=torch.float32, device=device)
    return o, lse


def check(o_gpu, lse_gpu, o_ref, lse_ref, what):
    o = o_gpu.float().cpu().numpy().astype(np.float64)
    lse = lse_gpu.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(o)), f"{what}: O not written or non-finite"
    if o.size:
        err = np.abs(o - o_ref)
        assert err.max() <= O_MAX, f"{what}: O max-abs {err.max():.3e}"
        assert err.mean() <= O_MEAN, f"{what}: O mean-abs {err.mean():.3e}"
    fin = np.isfinite(lse_ref)
    assert np.array_equal(np.isfinite(lse), fin), f"{what}: LSE finiteness differs"
    assert np.all(lse[~fin] == -np.inf), what
    if fin.any():
        lerr = np.abs(lse[fin] - lse_ref[fin]).max()
        assert lerr <= LSE_MAX, f"{what}: LSE max-abs {lerr:.3e}"


@pytest.mark.parametrize("i", range(24))
def test_random_prefill_batches(i):
    w = prefill_case(i)
    q, k, v = W.make_inputs(w, "cuda")
    o, lse = outputs(w, "cuda")
    pkg.opattn_prefill(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    torch.cuda.synchronize()
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    check(o, lse, o_ref, lse_ref, f"{w.name} (G {w.Hq // w.Hkv}, d {w.d}, Lq {w.q_lens}, Lk {w.k_lens})")


@pytest.mark.parametrize("i", range(16))
def test_random_decode_batches(i):
    w = decode_case(i)
    q, k, v = W.make_inputs(w, "cuda")
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    what = f"{w.name} (G {w.Hq // w.Hkv}, Lq {w.q_lens}, Lk {w.k_lens})"
    for name, call in (("prefill", pkg.opattn_prefill), ("decode", pkg.opattn_decode)):
        o, lse = outputs(w, "cuda")
        call(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
        torch.cuda.synchronize()
        check(o, lse, o_ref, lse_ref, f"{name} {what}")
