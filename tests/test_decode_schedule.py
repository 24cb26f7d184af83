"""Decode scheduler and argument checks of the decode entry points (no GPU).

Checked against brute-force enumeration: every (sequence, kv head, key tile)
is covered by exactly one chunk, chunks of a pair are contiguous and
numbered in tile order and sit on different CTAs, partial slots and merge
groups are unique and dense, and (stream-K cut) every CTA streams the same
number of key tiles to within one.  The default-grid schedule is checked for
the same cover, for one chunk per CTA on small batches and for the fitted
grid of a large uniform batch.
"""
import ctypes

import numpy as np
import pytest

import paper_2608_13499_gb300 as pkg
from paper_2608_13499_gb300 import build as pbuild

BN = 128


@pytest.fixture(scope="module", autouse=True)
def lib():
    pbuild.build()
    return pkg.load()


def table(units):
    return {name: units[:, i] for i, name in enumerate(pkg.DEC_UNIT_FIELDS)}


CASES = [
    # (q_lens, k_lens, Hq, Hkv, n_cta)
    ([1] * 9, [1, 2, 127, 128, 129, 255, 257, 1000, 3000], 16, 2, 152),
    ([2, 2, 2, 2], [5, 130, 700, 2049], 32, 8, 152),
    ([4, 4, 4, 4], [4, 64, 513, 4100], 16, 2, 7),
    ([3, 1, 0, 2], [1, 0, 5, 2], 16, 2, 152),            # Lq > Lk, no keys, no queries
    ([1, 1], [32768, 32768], 64, 8, 152),                 # long contexts are split
    ([1] * 64, [8192] * 64, 64, 8, 152),
    ([1], [40000], 8, 1, 1),                              # one CTA still splits into ~6 chunks
    ([1] * 5, [300, 9000, 17, 128 * 40, 1], 32, 1, 152),  # G = 32
]


def check_cover(lq, lk, Hkv, cu_q, cu_k, units, offs):
    """Every (sequence, kv head, key tile) in exactly one chunk; chunks numbered in tile order, one per CTA;
    partial slots contiguous per pair and dense; merge groups dense."""
    t = table(units)
    seen = {}
    for i in range(len(units)):
        s, h = int(t["seq"][i]), int(t["kvh"][i])
        assert lq[s] > 0
        assert t["q_tok0"][i] == cu_q[s] and t["nq"][i] == lq[s]
        assert t["k_row0"][i] == cu_k[s] and t["Lk"][i] == lk[s]
        seen.setdefault((s, h), []).append(i)
    want_pairs = {(s, h) for s in range(len(lq)) if lq[s] > 0 for h in range(Hkv)}
    assert set(seen) == want_pairs
    parts, groups = [], []
    for (s, h), idx in seen.items():
        n_t = (lk[s] + BN - 1) // BN
        idx = sorted(idx, key=lambda i: t["chunk"][i])
        n_chunks = len(idx)
        assert all(t["n_chunks"][i] == n_chunks for i in idx)
        assert [int(t["chunk"][i]) for i in idx] == list(range(n_chunks))
        covered = []
        for i in idx:
            covered += list(range(t["tile0"][i], t["tile0"][i] + t["n_tiles"][i]))
        assert covered == list(range(n_t))                   # contiguous, in order, exactly once
        cta_of = np.searchsorted(offs, np.arange(len(units)), side="right") - 1
        assert len({int(cta_of[i]) for i in idx}) == n_chunks           # one chunk per CTA
        if n_chunks == 1:
            assert t["part"][idx[0]] == -1 and t["group"][idx[0]] == -1
        else:
            g = {int(t["group"][i]) for i in idx}
            assert len(g) == 1 and -1 not in g
            groups.append(g.pop())
            p0 = int(t["part"][idx[0]])
            assert [int(t["part"][i]) for i in idx] == list(range(p0, p0 + n_chunks))
            parts += list(range(p0, p0 + n_chunks))
    assert sorted(groups) == list(range(len(groups)))
    assert sorted(parts) == list(range(len(parts)))
    assert offs[-1] == len(units)
    return t


@pytest.mark.parametrize("case", CASES)
def test_chunks_cover_every_key_tile_once(case):
    lq, lk, Hq, Hkv, n_cta = case
    cu_q = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    cu_k = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    units, offs = pkg.opattn_decode_schedule(cu_q, cu_k, Hq, Hkv, 128, n_cta)
    t = check_cover(lq, lk, Hkv, cu_q, cu_k, units, offs)
    # every CTA streams floor or ceil of the mean number of key tiles
    total = int(t["n_tiles"].sum())
    n_used = len(offs) - 1
    assert offs[-1] == len(units)
    if total > 0:
        assert n_used == min(n_cta, total)
        loads = np.array([t["n_tiles"][offs[c]:offs[c + 1]].sum() for c in range(n_used)])
        assert loads.min() >= total // n_used and loads.max() <= -(-total // n_used)


@pytest.mark.parametrize("case", CASES)
def test_default_grid_schedule_covers_every_key_tile_once(case):
    lq, lk, Hq, Hkv, sms = case
    cu_q = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    cu_k = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    units, offs = pkg.opattn_decode_schedule_default(cu_q, cu_k, Hq, Hkv, 128, sms)
    check_cover(lq, lk, Hkv, cu_q, cu_k, units, offs)
    assert 1 <= len(offs) - 1 <= sms


def default_schedule(B, L, sms=152, Hq=64, Hkv=8):
    cu_q = np.arange(B + 1, dtype=np.int32)
    cu_k = (cu_q * L).astype(np.int32)
    units, offs = pkg.opattn_decode_schedule_default(cu_q, cu_k, Hq, Hkv, 128, sms)
    t = check_cover([1] * B, [L] * B, Hkv, cu_q, cu_k, units, offs)
    return t, offs


@pytest.mark.parametrize("B,L,ctas,chunks", [
    (4, 1248, 128, {4}),     # 32 pairs of 10 tiles: 4 chunks of 2-3 tiles each, not 5-6 stream-K pieces
    (12, 1500, 96, {1}),     # 96 pairs of 12 tiles: one CTA each, nothing split
    (16, 2048, 128, {1}),    # 128 pairs of 16 tiles: one CTA each
    (1, 6268, 136, {17}),    # 8 pairs of 49 tiles: 17 chunks of at most 3 tiles
])
def test_small_batches_get_one_chunk_per_cta(B, L, ctas, chunks):
    """At most as many (sequence, kv head) pairs as SMs: the default grid cuts pair by pair, so no CTA
    holds the end of one split pair and the start of the next (about 3.8 us more on GB300)."""
    t, offs = default_schedule(B, L)
    assert len(offs) - 1 == ctas
    assert np.all(np.diff(offs) == 1)                       # one unit per CTA
    assert set(int(c) for c in t["n_chunks"]) == chunks
    n_t = -(-L // BN)
    m = -(-n_t // max(chunks))
    assert t["n_tiles"].max() == m and t["n_tiles"].min() >= n_t // max(chunks)


def test_large_uniform_batch_keeps_the_fitted_stream_k_grid():
    t, offs = default_schedule(64, 8192)                    # 512 pairs > 152 SMs
    assert len(offs) - 1 == 128 and set(int(c) for c in t["n_chunks"]) == {1}
    loads = np.array([t["n_tiles"][offs[c]:offs[c + 1]].sum() for c in range(128)])
    assert loads.min() == loads.max() == 4 * 64


def test_long_contexts_are_split_for_parallelism():
    units, offs = pkg.opattn_decode_schedule([0, 1, 2], [0, 32768, 65536], 64, 8, 128, 152)
    t = table(units)
    # 2 x 8 pairs of 256 tiles over 152 CTAs (26.9 tiles each): every pair spans about ten CTAs
    assert len(offs) == 153 and set(t["n_chunks"]) <= {10, 11}
    # one CTA: nothing is split
    units, offs = pkg.opattn_decode_schedule([0, 1, 2], [0, 32768, 65536], 64, 8, 128, 1)
    assert len(offs) == 2 and set(table(units)["n_chunks"]) == {1}


A = 0x10000


@pytest.mark.parametrize("kwargs,status", [
    (dict(d=64), pkg.OPATTN_ERR_UNSUPPORTED),                          # decode kernel is d = 128 only
    (dict(Hq=6, Hkv=2), pkg.OPATTN_ERR_UNSUPPORTED),                   # G = 3 does not divide 32
    (dict(Hq=64, Hkv=1), pkg.OPATTN_ERR_UNSUPPORTED),                  # G = 64 > 32 columns
    (dict(cu_q=(0, 5), cu_k=(0, 9)), pkg.OPATTN_ERR_UNSUPPORTED),      # 5 tokens x G 8 > 32 columns
    (dict(Hq=6, Hkv=4), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(q=A + 8), pkg.OPATTN_ERR_MISALIGNED),
    (dict(lse=None), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(scale=0.0), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(cu_q=(0, 0), cu_k=(0, 7)), pkg.OPATTN_OK),                   # no query rows: nothing to do
])
def test_decode_argument_errors(kwargs, status):
    args = dict(q=A, k=A, v=A, o=A, lse=A, cu_q=(0, 1), cu_k=(0, 9), n_seq=1, Hq=16, Hkv=2, d=128, scale=0.125)
    args.update(kwargs)
    st = pkg.opattn_decode(args["q"], args["k"], args["v"], args["o"], args["lse"], args["cu_q"], args["cu_k"],
                           args["n_seq"], args["Hq"], args["Hkv"], args["d"], args["scale"], stream=0, check=False)
    assert st == status


def test_decode_plan_and_schedule_validate():
    with pytest.raises(pkg.OpattnError) as e:
        pkg.Plan((0, 1), (0, 9), 16, 2, 64, decode=True)
    assert e.value.status == pkg.OPATTN_ERR_UNSUPPORTED
    lib = pkg.load()
    cu = np.array([0, 1], dtype=np.int32)
    n_units, n_used = ctypes.c_int64(0), ctypes.c_int32(0)
    st = lib.opattn_decode_schedule(cu.ctypes.data_as(ctypes.c_void_p), cu.ctypes.data_as(ctypes.c_void_p), 1,
                                    16, 2, 128, 0, None, 0, None, ctypes.byref(n_units), ctypes.byref(n_used))
    assert st == pkg.OPATTN_ERR_INVALID_ARG                             # n_ctas must be positive
    st = lib.opattn_decode_schedule_default(cu.ctypes.data_as(ctypes.c_void_p), cu.ctypes.data_as(ctypes.c_void_p),
                                            1, 16, 2, 128, 0, None, 0, None, ctypes.byref(n_units),
                                            ctypes.byref(n_used))
    assert st == pkg.OPATTN_ERR_INVALID_ARG                             # sms must be positive
    st = lib.opattn_decode_schedule_default(cu.ctypes.data_as(ctypes.c_void_p), cu.ctypes.data_as(ctypes.c_void_p),
                                            1, 16, 2, 64, 152, None, 0, None, ctypes.byref(n_units),
                                            ctypes.byref(n_used))
    assert st == pkg.OPATTN_ERR_UNSUPPORTED                             # the decode kernel is d = 128 only
    assert pkg.opattn_decode_checked(A, A, A, A, A, (0, 1), (0, 9), 1, 16, 2, 128, 0.1, stream=0,
                                     flags=0x40) == pkg.OPATTN_ERR_INVALID_ARG


@pytest.mark.parametrize("kwargs,status", [
    (dict(block_size=12), pkg.OPATTN_ERR_UNSUPPORTED),
    (dict(block_size=4), pkg.OPATTN_ERR_UNSUPPORTED),
    (dict(block_size=256), pkg.OPATTN_ERR_UNSUPPORTED),
    (dict(max_blocks=1), pkg.OPATTN_ERR_INVALID_ARG),          # 9 keys need 2 pages of 8
    (dict(max_blocks=0), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(seqlens_k=(-1,)), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(d=64), pkg.OPATTN_ERR_UNSUPPORTED),
    (dict(k=None), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(table=None), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(num_blocks=0), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(table=A + 2), pkg.OPATTN_ERR_MISALIGNED),
    (dict(v=A + 8), pkg.OPATTN_ERR_MISALIGNED),
    (dict(seqlens_k=(0,), q=None), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(cu_q=(0, 0)), pkg.OPATTN_OK),                         # no query rows: nothing to do
])
def test_paged_argument_errors(kwargs, status):
    args = dict(q=A, k=A, v=A, table=A, num_blocks=4, block_size=8, max_blocks=2, o=A, lse=A, cu_q=(0, 1),
                seqlens_k=(9,), Hq=16, Hkv=2, d=128, scale=0.125)
    args.update(kwargs)
    st = pkg.opattn_decode_paged(args["q"], args["k"], args["v"], args["table"], args["num_blocks"],
                                 args["block_size"], args["max_blocks"], args["o"], args["lse"], args["cu_q"],
                                 args["seqlens_k"], 1, args["Hq"], args["Hkv"], args["d"], args["scale"], stream=0,
                                 check=False)
    assert st == status


@pytest.mark.parametrize("kwargs,status", [
    (dict(block_size=12), pkg.OPATTN_ERR_UNSUPPORTED),
    (dict(max_blocks=1), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(d=96), pkg.OPATTN_ERR_UNSUPPORTED),
    (dict(k=None), pkg.OPATTN_ERR_INVALID_ARG),
    (dict(table=A + 2), pkg.OPATTN_ERR_MISALIGNED),
    (dict(cu_q=(0, 0)), pkg.OPATTN_OK),
])
def test_paged_prefill_argument_errors(kwargs, status):
    args = dict(q=A, k=A, v=A, table=A, num_blocks=4, block_size=8, max_blocks=2, o=A, lse=A, cu_q=(0, 5),
                seqlens_k=(9,), Hq=16, Hkv=2, d=128, scale=0.125)
    args.update(kwargs)
    st = pkg.opattn_prefill_paged(args["q"], args["k"], args["v"], args["table"], args["num_blocks"],
                                  args["block_size"], args["max_blocks"], args["o"], args["lse"], args["cu_q"],
                                  args["seqlens_k"], 1, args["Hq"], args["Hkv"], args["d"], args["scale"],
                                  stream=0, check=False)
    assert st == status


@pytest.mark.parametrize("seed", range(40))
def test_default_grid_schedule_on_random_batches(seed):
    """Seeded random ragged batches (empty sequences, Lq = 0, few and many pairs, 1 to 152 SMs): the
    default-grid schedule covers every key tile exactly once, uses at most the SMs given, and when it
    cuts pair by pair gives every CTA one chunk with keys."""
    rng = np.random.default_rng(500 + seed)
    G = int(rng.choice([1, 2, 4, 8, 16, 32]))
    Hkv = int(rng.choice([1, 2, 4, 8]))
    n_seq = int(rng.integers(1, 40))
    max_q = 32 // G
    lq = [int(rng.integers(0, max_q + 1)) for _ in range(n_seq)]
    lk = [int(rng.integers(0, 20000)) if rng.random() < 0.9 else 0 for _ in range(n_seq)]
    sms = int(rng.choice([1, 7, 64, 100, 152]))
    cu_q = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    cu_k = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    units, offs = pkg.opattn_decode_schedule_default(cu_q, cu_k, G * Hkv, Hkv, 128, sms)
    if len(units) == 0:
        assert sum(lq) == 0
        return
    t = check_cover(lq, lk, Hkv, cu_q, cu_k, units, offs)
    n_used = len(offs) - 1
    assert 1 <= n_used <= sms
    with_keys = np.array([int((t["n_tiles"][offs[c]:offs[c + 1]] > 0).sum()) for c in range(n_used)])
    pairs = sum(Hkv for s in range(n_seq) if lq[s] > 0 and lk[s] > 0)
    if 0 < pairs <= sms and with_keys.max() == 1:
        # pair-aligned: chunks of one pair differ by at most one tile
        for (s, h) in {(int(a), int(b)) for a, b in zip(t["seq"], t["kvh"])}:
            sizes = t["n_tiles"][(t["seq"] == s) & (t["kvh"] == h)]
            assert sizes.max() - sizes.min() <= 1
