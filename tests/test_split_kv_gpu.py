"""GPU parity of split-KV prefill: work units over long key ranges cut into pieces.

A batch of few prompt chunks over long cached prefixes (chunked prefill) has
fewer work units than SMs, so the scheduler cuts the units' key tiles into one
equal stretch per CTA.  Each piece writes a partial (O, LSE) and the piece that
finishes last merges them inside the same launch.  Every output element is
compared with the fp64 oracle (same bar as the other parity tests), and each
test first checks that its batch really is split on this GPU.
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


def sms():
    return torch.cuda.get_device_properties(0).multi_processor_count


def n_pieces(w, n_cta=None):
    units, _ = pkg.opattn_schedule(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, n_cta or sms())
    return int((units[:, pkg.UNIT_FIELDS.index("part")] >= 0).sum())


def outputs(w):
    o = torch.full((w.total_q, w.Hq, w.d), float("nan"), dtype=torch.bfloat16, device="cuda")
    lse = torch.full((w.total_q, w.Hq), float("nan"), dtype=torch.float32, device="cuda")
    return o, lse


def run_gpu(w, q, k, v):
    o, lse = outputs(w)
    pkg.opattn_prefill(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
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


def reference(w, q, k, v):
    return oracle.attention(q.cpu(), k.cpu(), v.cpu(), w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, w.scale)


def custom(name, lq, lk, Hq, Hkv, d, seed=0, input_scale=1.0):
    return W.Workload(name, list(lq), list(lk), Hq, Hkv, d, input_scale, seed)


CASES = [
    W.chunk_long_prefix(),                                                  # 1 x 512 over 16K, G = 4
    W.chunks_long_prefix(),                                                 # 4 x 512 over 8-16K
    custom("split_g8_d64_empty", [64, 0, 300], [20000, 5, 3000], 16, 2, 64, seed=1),
    custom("split_g3_short_kv", [9, 40, 5], [12000, 24000, 2], 12, 4, 128, seed=2),  # G = 3; Lq > Lk rows
    custom("split_g16", [100, 7], [12000, 9000], 32, 2, 128, seed=3),
    custom("split_g1", [130], [40000], 4, 4, 128, seed=4),
]


@pytest.mark.parametrize("w", CASES, ids=[w.name for w in CASES])
def test_split_units_every_element(w):
    assert n_pieces(w) > 0, "the batch is split on this GPU"
    q, k, v = W.make_inputs(w, "cuda")
    o, lse = run_gpu(w, q, k, v)
    o_ref, lse_ref = reference(w, q, k, v)
    check(o, lse, o_ref, lse_ref, w.name)


def test_growing_logits_across_pieces():
    """Logits grow along the key range (by ~0.002 nats per key, ~78 nats over the range), so
    the pieces' partial LSEs differ by tens of nats and the merge weights span many octaves."""
    w = custom("split_growing", [64], [40000], 16, 4, 64, seed=9)
    assert n_pieces(w) > 0
    q, k, v = W.make_inputs(w, "cuda")
    pos = torch.arange(w.total_k, dtype=torch.float32, device="cuda")
    qf = q.float() * 0.1
    qf[:, :, 0] = 16.0
    kf = k.float() * 0.1
    kf[:, :, 0] = (pos / 1024.0)[:, None]
    q, k = qf.to(torch.bfloat16), kf.to(torch.bfloat16)
    o, lse = run_gpu(w, q, k, v)
    o_ref, lse_ref = reference(w, q, k, v)
    assert lse_ref.max() > 60.0
    check(o, lse, o_ref, lse_ref, w.name)


def test_plan_runs_graph_replays_and_budget():
    """A split plan is one launch per run that advances its own epoch: repeated runs and
    CUDA graph replays give the one-shot call's bits; an SM-capped plan matches the oracle."""
    w = W.chunk_long_prefix()
    q, k, v = W.make_inputs(w, "cuda")
    o1, l1 = run_gpu(w, q, k, v)
    o_ref, lse_ref = reference(w, q, k, v)
    check(o1, l1, o_ref, lse_ref, "one-shot")
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d) as plan:
        o, lse = outputs(w)
        for i in range(3):
            o.fill_(float("nan"))
            plan.run(q, k, v, o, lse, w.scale)
            torch.cuda.synchronize()
            assert torch.equal(o, o1) and torch.equal(lse, l1), f"run {i}"
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            plan.run(q, k, v, o, lse, w.scale)
        for i in range(3):
            o.fill_(float("nan"))
            lse.fill_(float("nan"))
            graph.replay()
            torch.cuda.synchronize()
            assert torch.equal(o, o1) and torch.equal(lse, l1), f"replay {i}"
    assert n_pieces(w, 20) > 0
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, max_ctas=20) as plan:
        assert plan.n_ctas == 20
        o, lse = outputs(w)
        plan.run(q, k, v, o, lse, w.scale)
        torch.cuda.synchronize()
    check(o, lse, o_ref, lse_ref, "20-CTA plan")


def test_plan_stays_correct_after_a_run_that_stopped_early():
    """CTA 0 gives up on a wait (test flag, ~20 ms) while the other CTAs finish their pieces,
    so merge counters are left part-counted; the launch epoch makes later runs ignore them."""
    w = W.chunk_long_prefix()
    q, k, v = W.make_inputs(w, "cuda")
    o_ref, lse_ref = reference(w, q, k, v)
    units, offs = pkg.opattn_schedule(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, sms())
    assert (units[offs[0]:offs[1], pkg.UNIT_FIELDS.index("part")] >= 0).any()  # CTA 0 holds a piece
    with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d) as plan:
        o, lse = outputs(w)
        st = plan.run_checked(q, k, v, o, lse, w.scale, flags=pkg.OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA)
        assert st == pkg.OPATTN_ERR_TIMEOUT
        for i in range(2):
            o.fill_(float("nan"))
            lse.fill_(float("nan"))
            assert plan.run_checked(q, k, v, o, lse, w.scale) == pkg.OPATTN_OK
            check(o, lse, o_ref, lse_ref, f"run {i} after the early stop")


@pytest.mark.parametrize("page", [16, 128])
def test_paged_cache_split_matches_packed(page):
    """The pieces read their key tiles through the block table from their own first tile."""
    w = W.chunks_long_prefix()
    q, k, v = W.make_inputs(w, "cuda")
    o1, l1 = run_gpu(w, q, k, v)
    lay = W.paged_layout(w.k_lens, page, seed=5)
    kc, vc = W.to_paged(k, w.k_lens, lay), W.to_paged(v, w.k_lens, lay)
    table = torch.from_numpy(lay.block_table).to("cuda")
    o2, l2 = outputs(w)
    pkg.opattn_prefill_paged(q, kc, vc, table, lay.num_blocks, lay.page_size, lay.max_blocks, o2, l2, w.cu_q,
                             np.asarray(w.k_lens, dtype=np.int32), w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2) and torch.equal(l1, l2)


def test_noalloc_runs_the_unsplit_schedule_within_tolerance():
    w = W.chunk_long_prefix()
    q, k, v = W.make_inputs(w, "cuda")
    o_ref, lse_ref = reference(w, q, k, v)
    o, lse = outputs(w)
    pkg.opattn_prefill_noalloc(q, k, v, o, lse, w.cu_q, w.cu_k, w.n_seq, w.Hq, w.Hkv, w.d, w.scale)
    torch.cuda.synchronize()
    check(o, lse, o_ref, lse_ref, "no-alloc")


def random_split_case(i):
    """Seeded random chunked-prefill batch that the scheduler cuts into pieces on a 152-SM GPU:
    1-4 chunks of 1-300 queries over 8K-40K-key prefixes, G in {1, 2, 3, 4, 8, 16}, d in {64, 128},
    2 or 4 kv heads.  Draws that the list schedule would keep whole are drawn again."""
    rng = np.random.default_rng(7000 + i)
    while True:
        n = int(rng.integers(1, 5))
        G = int(rng.choice([1, 2, 3, 4, 8, 16]))
        Hkv = int(rng.choice([2, 4]))
        d = int(rng.choice([64, 128]))
        lq = [int(x) for x in rng.integers(1, 301, n)]
        lk = [q + int(p) for q, p in zip(lq, rng.integers(8000, 40001, n))]
        w = custom(f"rand_split_{i}", lq, lk, G * Hkv, Hkv, d, seed=7000 + i)
        if n_pieces(w, 152) > 0:
            return w


@pytest.mark.parametrize("i", range(10))
def test_random_split_batches_every_element(i):
    w = random_split_case(i)
    if n_pieces(w) == 0:
        pytest.skip("this batch is not split on this GPU")
    q, k, v = W.make_inputs(w, "cuda")
    o, lse = run_gpu(w, q, k, v)
    o_ref, lse_ref = reference(w, q, k, v)
    check(o, lse, o_ref, lse_ref, w.name)
