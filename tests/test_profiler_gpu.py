"""Operator profile on the GPU: SM budget and sparse-sampling interpolation.

Sanity bars only (the measured accuracy is reported by the profiler's own
report): a smaller SM budget never makes the launch faster, an eighth of the
SMs makes a compute-bound batch several times slower, and an interpolated
profile from a handful of points predicts held-out points roughly.
"""
import numpy as np
import pytest

import paper_2608_13499_gb300 as pkg
from paper_2608_13499_gb300 import build as pbuild
from paper_2608_13499_gb300 import profiler as P
from paper_2608_13499_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    pbuild.build()
    return pkg.load()


def test_latency_falls_with_sm_budget():
    w = W.Workload("sm_budget_4x2048", [2048] * 4, [2048] * 4, 32, 8, 128)
    sms = P.n_sms()
    budgets = [P.ctas_for_share(f, sms) for f in (0.125, 0.25, 0.5, 1.0)]
    curve = P.sm_budget_curve(w, budgets, reps=5)
    assert [n for n, _ in curve] == budgets
    ms = [t for _, t in curve]
    for a, b in zip(ms, ms[1:]):
        assert b <= a * 1.05, curve
    assert ms[0] >= 4.0 * ms[-1], curve


def test_small_profile_predicts_held_out_points():
    acc = P.profile_accuracy(12, 8, seed=3, b_range=(1, 8), l_range=(128, 2048), reps=3)
    assert np.all(acc["measured"] > 0)
    assert acc["errors"]["mean"] < 0.25, acc["errors"]
    prof = acc["profile"]
    np.testing.assert_allclose(prof.predict(prof.coords), prof.times_ms, rtol=1e-9)


def test_small_decode_profile_and_budget():
    acc = P.profile_accuracy(12, 8, seed=4, key=P.decode_key(64, 8, 128), b_range=(1, 64), l_range=(256, 8192),
                             reps=3)
    assert np.all(acc["measured"] > 0)
    assert acc["errors"]["mean"] < 0.25, acc["errors"]
    w = W.DECODE["decode_llama3_70b"]()
    sms = P.n_sms()
    curve = P.sm_budget_curve(w, [P.ctas_for_share(0.25, sms), sms], reps=3, decode=True)
    assert curve[0][1] > curve[1][1]          # a quarter of the SMs cannot stream as fast as all of them


def test_colocated_operators_share_the_gpu():
    """Prefill and decode on disjoint SM budgets run at once and give the same bits as alone."""
    import torch
    wa = W.Workload("coloc_prefill_4x1024", [1024] * 4, [1024] * 4, 32, 8, 128, 1.0, 21)
    wb = W.Workload("coloc_decode_16x4096", [1] * 16, [4096] * 16, 64, 8, 128, 1.0, 22)
    sms = P.n_sms()
    nb = P.ctas_for_share(0.25, sms)
    r = P.colocate(wa, wb, sms - nb, nb, span_ms=2.0, reps=2)
    assert r["ctas"] == (sms - nb, nb)
    assert all(t > 0 for t in r["alone_ms"] + r["colocated_ms"] + r["full_gpu_ms"])
    assert r["makespan_ms"] > 0 and r["speedup"] > 0
    assert all(i > 0 for i in r["interference"])
    # outputs of co-located launches equal those of the same plans run alone
    outs = {}
    for mode in ("alone", "together"):
        s_a, s_b = torch.cuda.Stream(), torch.cuda.Stream()
        res = []
        plans = []
        for w, dec, n, s in ((wa, False, sms - nb, s_a), (wb, True, nb, s_b)):
            q, k, v = W.make_inputs(w, "cuda")
            o = torch.full((w.total_q, w.Hq, w.d), float("nan"), dtype=torch.bfloat16, device="cuda")
            lse = torch.full((w.total_q, w.Hq), float("nan"), dtype=torch.float32, device="cuda")
            plans.append((pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, max_ctas=n, decode=dec), (q, k, v, o, lse, w.scale), s))
            res.append((o, lse))
        torch.cuda.synchronize()
        for plan, args, s in plans:
            plan.run(*args, s)
            if mode == "alone":
                s.synchronize()
        torch.cuda.synchronize()
        for plan, _, _ in plans:
            plan.close()
        outs[mode] = [(o.clone(), lse.clone()) for o, lse in res]
    for (oa, la), (ob, lb) in zip(outs["alone"], outs["together"]):
        assert torch.isfinite(oa.float()).all()
        assert torch.equal(oa, ob) and torch.equal(la, lb)
