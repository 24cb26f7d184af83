"""GPU parity of the decode kernel (opattn_decode, through the C ABI) against the fp64 oracle.

Same bar as the prefill kernel: O within max-abs 1e-2 and mean-abs 1e-3,
LSE within 1e-3 where the oracle's is finite and exactly -inf where not.
The oracle is the same attention definition: decode rows are causal rows
whose query sits at the end of the sequence.  Cases cover one and several
query tokens per sequence, G from 1 to 32, key counts around the 128-key
tile edges, sequences without keys or queries and with Lq > Lk, key ranges
split into many chunks (and the same batch split differently), scores that
move the softmax base across tiles, and the full-size decode workloads on
sampled rows.
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


def run_decode(w, q, k, v, max_ctas=None, stream=None):
    o = torch.full((w.total_q, w.Hq, w.d), float("nan"), dtype=torch.bfloat16, device=q.device)
    lse = torch.full((w.total_q, w.Hq), float("nan"), dtype=torch.float32, device=q.device)
    if max_ctas is None:
        pkg.opattn_decode(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale, stream)
    else:
        with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, max_ctas=max_ctas, decode=True) as plan:
            plan.run(q, k, v, o, lse, w.scale, stream)
            torch.cuda.synchronize()
    torch.cuda.synchronize()
    return o, lse


def check(o_gpu, lse_gpu, o_ref, lse_ref, what=""):
    o = o_gpu.float().cpu().numpy().astype(np.float64)
    lse = lse_gpu.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(o)), f"{what}: non-finite O (unwritten rows?)"
    err = np.abs(o - o_ref)
    assert err.max() <= O_MAX, f"{what}: O max-abs {err.max():.3e}"
    assert err.mean() <= O_MEAN, f"{what}: O mean-abs {err.mean():.3e}"
    fin = np.isfinite(lse_ref)
    assert np.array_equal(np.isfinite(lse), fin), f"{what}: LSE finiteness differs"
    assert np.all(lse[~fin] == -np.inf)
    if fin.any():
        lerr = np.abs(lse[fin] - lse_ref[fin]).max()
        assert lerr <= LSE_MAX, f"{what}: LSE max-abs {lerr:.3e}"
    return err.max(), err.mean()


def custom(name, lq, lk, Hq, Hkv, seed=0, input_scale=1.0):
    return W.Workload(name, list(lq), list(lk), Hq, Hkv, 128, input_scale, seed)


SMALL = [
    custom("dec_g8_tile_edges", [1] * 9, [1, 2, 127, 128, 129, 255, 257, 1000, 3000], 16, 2),
    custom("dec_g4_two_tokens", [2] * 4, [5, 130, 700, 2049], 32, 8, seed=1),
    custom("dec_g8_four_tokens", [4] * 4, [4, 64, 513, 4100], 16, 2, seed=2),
    custom("dec_g1_mha", [1, 1, 1], [1, 300, 5000], 8, 8, seed=3),
    custom("dec_g32", [1, 1], [77, 1500], 32, 1, seed=4),
    custom("dec_g2_sixteen_tokens", [16, 3], [40, 900], 4, 2, seed=5),
    custom("dec_edges", [3, 1, 0, 2], [1, 0, 5, 2], 16, 2, seed=6),       # Lq > Lk, no keys, no queries
    custom("dec_long_split", [1, 2], [40000, 20000], 8, 1, seed=7),       # many chunks, in-kernel merge
    custom("dec_scaled_half", [1] * 6, [3000, 17, 900, 129, 4096, 60], 32, 8, seed=8, input_scale=0.5),
]


@pytest.mark.parametrize("w", SMALL, ids=[w.name for w in SMALL])
def test_small_cases_every_element(w):
    q, k, v = W.make_inputs(w, "cuda")
    o, lse = run_decode(w, q, k, v)
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    check(o, lse, o_ref, lse_ref, w.name)


@pytest.mark.parametrize("max_ctas", [1, 5, 152])
def test_split_choices_agree(max_ctas):
    """The same batch with 1, 5 and 152 CTAs is cut into different chunks; all match the oracle."""
    w = custom("dec_split_choices", [1, 1, 3], [9000, 2500, 6000], 16, 2, seed=11)
    q, k, v = W.make_inputs(w, "cuda")
    o, lse = run_decode(w, q, k, v, max_ctas=max_ctas)
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    check(o, lse, o_ref, lse_ref, f"max_ctas={max_ctas}")


def test_growing_scores_move_the_base():
    """Scores grow along the keys (~0.07 nats per key), so later tiles exceed a
    chunk's first-tile maximum by far more than the kernel's slack: the base
    moves and the running sums and the O accumulator are rescaled."""
    w = custom("dec_growing", [1, 2], [4096, 3000], 16, 2, seed=9)
    q, k, v = W.make_inputs(w, "cuda")
    pos = torch.cat([torch.arange(n, dtype=torch.float32) for n in w.k_lens]).to("cuda")
    qf = q.float() * 0.1
    qf[:, :, 0] = 24.0
    kf = k.float() * 0.1
    kf[:, :, 0] = (pos / 32.0)[:, None]
    q, k = qf.to(torch.bfloat16), kf.to(torch.bfloat16)
    for max_ctas in (None, 1):
        o, lse = run_decode(w, q, k, v, max_ctas=max_ctas)
        o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
        assert lse_ref.max() > 150.0
        check(o, lse, o_ref, lse_ref, f"growing max_ctas={max_ctas}")


def test_large_logits():
    w = custom("dec_large_logits", [1, 4], [2000, 700], 16, 2, seed=12)
    q, k, v = W.make_inputs(w, "cuda")
    q = (q.float() * 4).to(torch.bfloat16)
    o, lse = run_decode(w, q, k, v)
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    check(o, lse, o_ref, lse_ref, w.name)


def test_matches_prefill_kernel_on_the_same_batch():
    """The two kernels compute the same function: their outputs agree to rounding."""
    w = custom("dec_vs_prefill", [1, 3, 2], [5000, 260, 129], 32, 8, seed=13)
    q, k, v = W.make_inputs(w, "cuda")
    o_d, lse_d = run_decode(w, q, k, v)
    o_p = torch.empty_like(o_d)
    lse_p = torch.empty_like(lse_d)
    pkg.opattn_prefill(q, k, v, o_p, lse_p, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    torch.cuda.synchronize()
    assert (o_d.float() - o_p.float()).abs().max().item() <= 1e-2
    assert (lse_d - lse_p).abs().max().item() <= 1e-3


def test_plan_repeat_runs_on_a_side_stream():
    """Each completed run leaves the plan's merge counters at zero: repeated runs stay correct."""
    w = custom("dec_plan_repeat", [1, 1], [30000, 7000], 16, 2, seed=14)
    q, k, v = W.make_inputs(w, "cuda")
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    side = torch.cuda.Stream()
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=True) as plan:
        assert plan.n_units > w.Hkv * w.n_seq          # the key ranges are split
        o = torch.empty((w.total_q, w.Hq, w.d), dtype=torch.bfloat16, device="cuda")
        lse = torch.empty((w.total_q, w.Hq), dtype=torch.float32, device="cuda")
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            for _ in range(3):
                o.fill_(float("nan"))
                plan.run(q, k, v, o, lse, w.scale, side)
        side.synchronize()
        check(o, lse, o_ref, lse_ref, "plan x3")


def test_plan_run_replays_from_a_cuda_graph():
    """A decode plan run is one kernel launch that advances its own launch epoch (the merge
    counters are tagged with it), so a captured run replays correctly, over key ranges split
    into up to 19 chunks."""
    w = custom("dec_graph", [1, 1, 1], [6268, 512, 3000], 64, 8, seed=16)
    q, k, v = W.make_inputs(w, "cuda")
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=True) as plan:
        assert plan.n_units > 2 * w.Hkv * w.n_seq  # the key ranges are split
        o = torch.empty((w.total_q, w.Hq, w.d), dtype=torch.bfloat16, device="cuda")
        lse = torch.empty((w.total_q, w.Hq), dtype=torch.float32, device="cuda")
        plan.run(q, k, v, o, lse, w.scale)  # outside the capture: first-use set-up
        torch.cuda.synchronize()
        check(o, lse, o_ref, lse_ref, "eager")
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            plan.run(q, k, v, o, lse, w.scale)
        for i in range(4):
            o.fill_(float("nan"))
            lse.fill_(float("nan"))
            graph.replay()
            torch.cuda.synchronize()
            check(o, lse, o_ref, lse_ref, f"replay {i}")


def test_forced_timeout_reports_and_context_survives():
    w = custom("dec_timeout", [1], [1000], 16, 2, seed=15)
    q, k, v = W.make_inputs(w, "cuda")
    o = torch.empty((1, 16, 128), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((1, 16), dtype=torch.float32, device="cuda")
    st = pkg.opattn_decode_checked(q, k, v, o, lse, w.cu_q, w.cu_k, 1, 16, 2, 128, w.scale,
                                   flags=pkg.OPATTN_FLAG_TEST_FORCE_TIMEOUT)
    assert st == pkg.OPATTN_ERR_TIMEOUT
    assert pkg.opattn_decode_checked(q, k, v, o, lse, w.cu_q, w.cu_k, 1, 16, 2, 128, w.scale) == pkg.OPATTN_OK
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    check(o, lse, o_ref, lse_ref, "after timeout")


def test_plan_stays_correct_after_a_run_that_stopped_early():
    """CTA 0 of a plan run gives up on a wait (test flag, ~20 ms) while the other CTAs finish their
    chunks, so the split pairs' merge counters are left part-counted.  The counters carry the launch
    epoch, which the kernel advances, so the following runs of the same plan ignore those counts."""
    w = custom("dec_partial_abort", [1, 1, 1], [6268, 512, 3000], 64, 8, seed=17)
    q, k, v = W.make_inputs(w, "cuda")
    o_ref, lse_ref = oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=True) as plan:
        units, offs = pkg.opattn_decode_schedule_default(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d,
                                                         torch.cuda.get_device_properties(0).multi_processor_count)
        assert len(units) == plan.n_units
        first = units[offs[0]:offs[1]]
        assert (first[:, pkg.DEC_UNIT_FIELDS.index("n_chunks")] > 1).any()  # CTA 0 holds a chunk of a split pair
        o = torch.empty((w.total_q, w.Hq, w.d), dtype=torch.bfloat16, device="cuda")
        lse = torch.empty((w.total_q, w.Hq), dtype=torch.float32, device="cuda")
        st = plan.run_checked(q, k, v, o, lse, w.scale, flags=pkg.OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA)
        assert st == pkg.OPATTN_ERR_TIMEOUT
        for i in range(3):
            o.fill_(float("nan"))
            lse.fill_(float("nan"))
            assert plan.run_checked(q, k, v, o, lse, w.scale) == pkg.OPATTN_OK
            check(o, lse, o_ref, lse_ref, f"run {i} after the early stop")


@pytest.mark.parametrize("name", sorted(W.DECODE))
def test_full_size_workloads_on_sampled_rows(name):
    w = W.DECODE[name]()
    q, k, v = W.make_inputs(w, "cuda")
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=True) as plan:
        o = torch.full((w.total_q, w.Hq, w.d), float("nan"), dtype=torch.bfloat16, device="cuda")
        lse = torch.full((w.total_q, w.Hq), float("nan"), dtype=torch.float32, device="cuda")
        plan.run(q, k, v, o, lse, w.scale)
        torch.cuda.synchronize()
    assert torch.isfinite(o.float()).all().item() and not torch.isnan(lse).any().item()
    rng = np.random.default_rng(0)
    n = 48
    tok = rng.integers(0, w.total_q, n)
    hd = rng.integers(0, w.Hq, n)
    tok[:2], hd[:2] = [0, w.total_q - 1], [0, w.Hq - 1]
    o_r, lse_r = oracle.attention_rows(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale,
                                       tok, hd)
    check(o[tok, hd], lse[tok, hd], o_r, lse_r, name)


def test_default_grid_splits_no_pair_of_a_uniform_batch():
    # 64 requests x 8192 keys, 8 kv heads: 512 (sequence, kv head) pairs of 64 key tiles each
    w = W.DECODE["decode_llama3_70b"]()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    pairs = w.n_seq * w.Hkv
    fits = [n for n in range((sms * 4 + 4) // 5, sms + 1) if pairs % n == 0]
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=True) as plan:
        assert (sms * 4 + 4) // 5 <= plan.n_ctas <= sms
        if fits:
            assert plan.n_ctas == max(fits)
            assert plan.n_units == pairs  # whole pairs per CTA: nothing split, nothing merged
    # an explicit SM budget is kept as given
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=True, max_ctas=sms) as plan:
        assert plan.n_ctas == sms
    # a ragged batch keeps the full grid
    r = W.DECODE["decode_llama3_8b"]()
    with pkg.Plan(r.cu_q, r.cu_k, r.Hq, r.Hkv, r.d, decode=True) as plan:
        assert plan.n_ctas == sms
