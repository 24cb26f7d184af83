"""Host scheduler (L2-grouped ragged work list), checked without a GPU.

The unit records are checked against a brute-force enumeration of which
(query token, key) pairs the causal mask leaves visible, and the assignment
against a replay of its rules: (sequence, kv head) pairs gathered in order
into groups of at most 48 MB of K/V, units taken group by group and longest
first within a group, each given to the least-loaded CTA (list scheduling:
makespan within mean load + largest unit); or, when that makespan is set by
a few long units, the stream-K cut of all key tiles into one equal stretch
per CTA, with the units cut by stretch boundaries split into pieces.
"""
import numpy as np
import pytest

import paper_2608_13499_gb300 as pkg
from paper_2608_13499_gb300 import build as pbuild
from paper_2608_13499_gb300 import workloads as W

BN = 128


@pytest.fixture(scope="module", autouse=True)
def lib():
    pbuild.build()
    return pkg.load()


def unit_table(units):
    return {name: units[:, i] for i, name in enumerate(pkg.UNIT_FIELDS)}


CASES = [
    ([1, 17, 64], [1, 17, 64], 4, 2, 64, 152),
    ([1, 2, 127, 128, 129, 255, 257], [1, 2, 127, 128, 129, 255, 257], 32, 8, 128, 7),
    ([512, 512, 300], [700, 1024, 300], 32, 8, 128, 16),     # chunks with prefixes
    ([9, 0, 40, 5], [3, 0, 40, 0], 12, 4, 128, 5),            # Lq > Lk, empty, G = 3
    ([100, 33], [100, 33], 128, 1, 64, 3),                    # G = 128, one token per M-tile
    (W.bursty().q_lens, W.bursty().k_lens, 32, 8, 128, 152),
]


SPLIT_CASES = [
    ([512], [16896], 32, 8, 128, 152),                        # one chunk over a 16K prefix
    ([512, 512, 300], [9000, 17000, 12000], 32, 8, 128, 152),  # a few chunks over long prefixes
    ([64, 0, 2000], [40000, 5, 2000], 16, 2, 64, 100),        # G = 8, d = 64, an empty sequence
    ([5, 3], [3000, 1], 12, 4, 128, 8),                       # G = 3, Lq > Lk rows
]


@pytest.mark.parametrize("case", CASES + SPLIT_CASES)
def test_units_cover_every_row_once_with_exact_tile_counts(case):
    """Every (token, kv head) row is in exactly one unit, and the pieces of a split unit
    cover its key tiles [0, n_tiles) once, in order, with contiguous partial slots."""
    lq, lk, Hq, Hkv, d, n_cta = case
    cu_q = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    cu_k = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    units, offs = pkg.opattn_schedule(cu_q, cu_k, Hq, Hkv, d, n_cta)
    G = Hq // Hkv
    tpu = 2 * (128 // G)
    t = unit_table(units)
    covered = np.zeros((int(cu_q[-1]), Hkv), dtype=np.int32)
    pieces = {}
    for u in range(len(units)):
        s = t["seq"][u]
        L_q, L_k = lq[s], lk[s]
        delta = L_k - L_q
        tok0 = t["q_tok0"][u] - cu_q[s]
        assert 0 <= tok0 < L_q and tok0 % tpu == 0
        assert t["n_tok"][u] == min(tpu, L_q - tok0)
        assert t["k_row0"][u] == cu_k[s] and t["Lk"][u] == L_k
        assert t["qlim0"][u] == tok0 + delta
        pieces.setdefault((s, t["kvh"][u], tok0), []).append(u)
    slots, groups = set(), set()
    for (s, h, tok0), us in pieces.items():
        L_q, L_k = lq[s], lk[s]
        n_tok = min(tpu, L_q - tok0)
        covered[cu_q[s] + tok0:cu_q[s] + tok0 + n_tok, h] += 1
        # brute force: the highest key any token of the unit sees
        last = max([min(i + L_k - L_q, L_k - 1) for i in range(tok0, tok0 + n_tok)])
        want_tiles = 0 if last < 0 else last // BN + 1
        us = sorted(us, key=lambda u: t["chunk"][u])
        k = len(us)
        assert [t["chunk"][u] for u in us] == list(range(k))
        assert all(t["n_chunks"][u] == k for u in us)
        tiles = [(t["tile0"][u], t["n_tiles"][u]) for u in us]
        assert tiles[0][0] == 0 and sum(n for _, n in tiles) == want_tiles
        assert all(a0 + an == b0 for (a0, an), (b0, _) in zip(tiles, tiles[1:]))
        if k == 1:
            assert t["part"][us[0]] == -1 and t["group"][us[0]] == -1
        else:
            assert all(n > 0 for _, n in tiles)
            part0 = t["part"][us[0]]
            assert [t["part"][u] for u in us] == list(range(part0, part0 + k))
            assert len({t["group"][u] for u in us}) == 1
            slots.update(range(part0, part0 + k))
            groups.add(t["group"][us[0]])
    assert np.all(covered == 1)
    assert slots == set(range(len(slots))) and groups == set(range(len(groups)))
    if case in SPLIT_CASES:
        assert groups, "a batch of few long units is split"


GROUP_BYTES = 48 << 20


def expected_order(lq, lk, Hkv, d, G):
    """(group, unit) keys in the order the scheduler assigns units."""
    tpu = 2 * (128 // G)
    keys, group, gbytes = [], 0, 0
    for s in range(len(lq)):
        if lq[s] == 0:
            continue
        for h in range(Hkv):
            pb = lk[s] * 2 * d * 2
            if gbytes > 0 and gbytes + pb > GROUP_BYTES:
                group, gbytes = group + 1, 0
            gbytes += pb
            for t0 in range(0, lq[s], tpu):
                n_tok = min(tpu, lq[s] - t0)
                last = min(t0 + lk[s] - lq[s] + n_tok - 1, lk[s] - 1)
                n_tiles = 0 if last < 0 else last // BN + 1
                keys.append((group, n_tiles, s, h, t0))
    # stable: group ascending, tiles descending
    return sorted(keys, key=lambda k: (k[0], -k[1]))


def random_cases(n, seed=123):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        Hkv = int(rng.choice([1, 2, 8]))
        G = int(rng.choice([1, 3, 4, 8, 16]))
        d = int(rng.choice([64, 128]))
        n_seq = int(rng.integers(1, 12))
        lq = [int(x) for x in rng.integers(0, 3000, n_seq)]
        lk = [max(0, q + int(rng.integers(-50, 9000))) for q in lq]
        out.append((lq, lk, G * Hkv, Hkv, d, int(rng.choice([1, 5, 64, 152, 1000]))))
    return out


# The last case's loads span more buckets than the bucket queue takes
# (1024 CTAs x 70K-tile units), so the scheduler uses its heap there.
SPLIT_GAIN = 0.85  # the cut replaces the list schedule below this fraction of its makespan
PIECE_OVERHEAD = 2
MIN_STRETCH = 4    # ... and only when a CTA's stretch has at least this many key tiles


def list_schedule(order, n_cta):
    import heapq
    P = min(n_cta, len(order))
    heap = [(0, c) for c in range(P)]
    per_cta = [[] for _ in range(P)]
    for grp, n_tiles, s, h, t0 in order:
        load, c = heapq.heappop(heap)
        per_cta[c].append((s, h, t0, n_tiles, 0, -1, -1, 0, 1))
        heapq.heappush(heap, (load + n_tiles + 1, c))
    return per_cta


def stream_k_schedule(order, n_cta):
    """The cut of all key tiles, units in pair order, into one equal stretch per CTA."""
    units = sorted(order, key=lambda k: (k[2], k[3], k[4]))  # pair order: sequence, kv head, block
    total = sum(u[1] for u in units)
    P = max(1, min(n_cta, total))
    bound = lambda c: c * total // P  # noqa: E731
    per_cta = [[] for _ in range(P)]
    pos, rr, parts, groups = 0, 0, 0, 0
    for grp, n_tiles, s, h, t0 in units:
        if n_tiles <= 0:
            per_cta[rr].append((s, h, t0, 0, 0, -1, -1, 0, 1))
            rr = (rr + 1) % P
            continue
        c = next(c for c in range(P) if bound(c) <= pos < (bound(c + 1) if c + 1 < P else total + 1))
        pieces, t, end = [], pos, pos + n_tiles
        while t < end:
            stop = min(end, bound(c + 1)) if c + 1 < P else end
            if stop > t:
                pieces.append((c, t - pos, stop - t))
            t, c = stop, c + 1
        k = len(pieces)
        for i, (cc, a, n) in enumerate(pieces):
            per_cta[cc].append((s, h, t0, n, a, parts + i if k > 1 else -1, groups if k > 1 else -1, i, k))
        if k > 1:
            parts, groups = parts + k, groups + 1
        pos = end
    return per_cta


def makespan(per_cta):
    return max(sum(u[3] + 1 + (PIECE_OVERHEAD if u[5] >= 0 else 0) for u in us) for us in per_cta)


@pytest.mark.parametrize("case", CASES + [(W.chunked().q_lens, W.chunked().k_lens, 32, 8, 128, 152)] +
                         random_cases(24) + [([512000], [9000000], 1, 1, 64, 1024)] + SPLIT_CASES)
def test_group_major_list_assignment(case):
    """Replays both schedules and the choice between them, and compares unit by unit."""
    lq, lk, Hq, Hkv, d, n_cta = case
    cu_q = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    cu_k = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    units, offs = pkg.opattn_schedule(cu_q, cu_k, Hq, Hkv, d, n_cta)
    G = Hq // Hkv
    order = expected_order(lq, lk, Hkv, d, G)
    if len(order) == 0:
        assert len(units) == 0
        return
    want = list_schedule(order, n_cta)
    lpt = makespan(want)
    total = sum(u[1] + 1 for u in order)
    tiles = sum(u[1] for u in order)
    if tiles >= MIN_STRETCH * n_cta and lpt * SPLIT_GAIN > total / n_cta:
        sk = stream_k_schedule(order, n_cta)
        if makespan(sk) < SPLIT_GAIN * lpt:
            want = sk
    P = len(offs) - 1
    assert P == len(want)
    assert offs[0] == 0 and offs[-1] == len(units) and np.all(np.diff(offs) >= 1)
    t = unit_table(units)
    for c in range(P):
        got = [(int(t["seq"][i]), int(t["kvh"][i]), int(t["q_tok0"][i] - cu_q[t["seq"][i]]), int(t["n_tiles"][i]),
                int(t["tile0"][i]), int(t["part"][i]), int(t["group"][i]), int(t["chunk"][i]), int(t["n_chunks"][i]))
               for i in range(offs[c], offs[c + 1])]
        assert got == want[c], f"CTA {c}"
    if (t["part"] < 0).all():  # the list schedule's bound
        cost = t["n_tiles"].astype(np.int64) + 1
        loads = np.array([cost[offs[c]:offs[c + 1]].sum() for c in range(P)])
        assert loads.max() <= cost.sum() / P + cost.max() + 1e-9


def test_standard_workloads_are_not_split():
    for w in [W.llama3_8b(), W.llama3_70b(), W.bursty(), W.chunked(), W.tiny()]:
        units, _ = pkg.opattn_schedule(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, 152)
        assert (units[:, pkg.UNIT_FIELDS.index("part")] == -1).all(), w.name


def test_small_batches_are_not_split():
    """Fewer key tiles than 4 per CTA: the list schedule is kept whatever its makespan."""
    for lq, lk, Hq, Hkv, d in [([300, 45, 129], [300, 45, 129], 16, 4, 128),
                               ([300, 1, 129, 700], [300, 1, 129, 700], 8, 2, 64),
                               ([300, 1, 129, 700], [300, 1, 129, 700], 8, 8, 64)]:
        cu_q = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
        cu_k = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
        units, _ = pkg.opattn_schedule(cu_q, cu_k, Hq, Hkv, d, 152)
        assert (units[:, pkg.UNIT_FIELDS.index("part")] == -1).all()


def test_groups_keep_each_groups_kv_within_l2():
    """Llama-3-70B layer: 64 pairs of 2 MB K/V -> groups of 24 pairs (48 MB); every CTA's units visit
    the groups in order, so the whole GPU works through one group's K/V at a time."""
    w = W.llama3_70b()
    units, offs = pkg.opattn_schedule(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, 152)
    t = unit_table(units)
    pair = t["seq"] * w.Hkv + t["kvh"]
    group = pair // 24
    for c in range(len(offs) - 1):
        assert np.all(np.diff(group[offs[c]:offs[c + 1]]) >= 0)


def test_capacity_error_reports_the_needed_size():
    cu = np.array([0, 300], dtype=np.int32)
    lib = pkg.load()
    import ctypes
    n_units, n_used = ctypes.c_int64(0), ctypes.c_int32(0)
    units = np.zeros((2, len(pkg.UNIT_FIELDS)), dtype=np.int32)
    offs = np.zeros(8, dtype=np.int32)
    st = lib.opattn_schedule(cu.ctypes.data_as(ctypes.c_void_p), cu.ctypes.data_as(ctypes.c_void_p), 1, 8, 2, 128, 4,
                             units.ctypes.data_as(ctypes.c_void_p), 2, offs.ctypes.data_as(ctypes.c_void_p),
                             ctypes.byref(n_units), ctypes.byref(n_used))
    assert st == pkg.OPATTN_ERR_CAPACITY
    # G = 4 -> 64 tokens per unit -> 5 blocks x 2 kv heads
    assert n_units.value == 10 and n_used.value == 4


def test_standard_workload_unit_counts():
    # G = 8 (Llama-3-70B shape): 32 tokens per unit -> 8 * 128 blocks * 8 kv heads
    w = W.llama3_70b()
    units, _ = pkg.opattn_schedule(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, 152)
    assert len(units) == 8 * 128 * 8
    w = W.tiny()
    units, _ = pkg.opattn_schedule(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, 152)
    assert len(units) == 6


def test_opattn_log_prints_work_list_statistics():
    """OPATTN_LOG=1 makes every schedule print one line on stderr: units, CTAs, largest and
    mean CTA load, largest unit, host time (checked on the host-only scheduler)."""
    import re
    import subprocess
    import sys
    code = ("import paper_2608_13499_gb300 as pkg\n"
            "units, offs = pkg.opattn_schedule([0, 300, 700], [0, 300, 900], 32, 8, 128, 5)\n"
            "cost = units[:, 6].astype(int) + 1\n"
            "loads = [int(cost[offs[c]:offs[c + 1]].sum()) for c in range(len(offs) - 1)]\n"
            "print(len(units), len(offs) - 1, max(loads), sum(loads), int(cost.max()))\n")
    env = dict(__import__("os").environ, OPATTN_LOG="1")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, check=True)
    n, n_cta, mx, total, biggest = map(int, r.stdout.split())
    lines = [ln for ln in r.stderr.splitlines() if ln.startswith("opattn:")]
    assert len(lines) == 2  # the binding asks for the size first, then for the list
    m = re.match(r"opattn: prefill schedule: (\d+) units on (\d+) CTAs; CTA load max (\d+) mean ([\d.]+) "
                 r"\(max/mean ([\d.]+)\); largest unit (\d+); host ([\d.]+) us", lines[-1])
    assert m, lines[-1]
    assert int(m.group(1)) == n and int(m.group(2)) == n_cta and int(m.group(3)) == mx
    assert abs(float(m.group(4)) - total / n_cta) < 0.05 and int(m.group(6)) == biggest
    env["OPATTN_LOG"] = "0"
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, check=True)
    assert "opattn:" not in r.stderr


def test_repeated_schedules_on_one_thread_are_identical():
    """The scheduler keeps its working arrays per host thread and reuses them: a list built after
    larger and smaller ones (arrays grown, then partly reused) must equal the one built first."""
    shapes = [
        (W.llama3_8b().q_lens, W.llama3_8b().k_lens, 32, 8, 128, 152),
        (W.bursty().q_lens, W.bursty().k_lens, 32, 8, 128, 152),   # larger: the arrays grow
        ([1, 17, 64], [1, 17, 64], 4, 2, 64, 152),                 # smaller: stale tails remain
        ([512], [16896], 32, 8, 128, 152),                         # the split-KV cut
    ]
    def sched(shape):
        lq, lk, Hq, Hkv, d, n_cta = shape
        cu_q = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
        cu_k = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
        return pkg.opattn_schedule(cu_q, cu_k, Hq, Hkv, d, n_cta)
    first = [sched(s) for s in shapes]
    for s, (u0, o0) in reversed(list(zip(shapes, first))):
        u1, o1 = sched(s)
        assert np.array_equal(u0, u1) and np.array_equal(o0, o1)
