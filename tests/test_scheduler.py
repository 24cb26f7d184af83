"""Host scheduler (L2-grouped ragged work list), checked without a GPU.

The unit records are checked against a brute-force enumeration of which
(query token, key) pairs the causal mask leaves visible, and the assignment
against a replay of its rule: (sequence, kv head) pairs gathered in order
into groups of at most 48 MB of K/V, units taken group by group and longest
first within a group, each given to the least-loaded CTA (list scheduling:
makespan within mean load + largest unit).
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


@pytest.mark.parametrize("case", CASES)
def test_units_cover_every_row_once_with_exact_tile_counts(case):
    lq, lk, Hq, Hkv, d, n_cta = case
    cu_q = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    cu_k = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    units, offs = pkg.opattn_schedule(cu_q, cu_k, Hq, Hkv, d, n_cta)
    G = Hq // Hkv
    tpu = 2 * (128 // G)
    t = unit_table(units)
    covered = np.zeros((int(cu_q[-1]), Hkv), dtype=np.int32)
    for u in range(len(units)):
        s = t["seq"][u]
        L_q, L_k = lq[s], lk[s]
        delta = L_k - L_q
        tok0 = t["q_tok0"][u] - cu_q[s]
        assert 0 <= tok0 < L_q and tok0 % tpu == 0
        assert t["n_tok"][u] == min(tpu, L_q - tok0)
        assert t["k_row0"][u] == cu_k[s] and t["Lk"][u] == L_k
        assert t["qlim0"][u] == tok0 + delta
        covered[t["q_tok0"][u]:t["q_tok0"][u] + t["n_tok"][u], t["kvh"][u]] += 1
        # brute force: the highest key any token of the unit sees
        last = max([min(i + delta, L_k - 1) for i in range(tok0, tok0 + t["n_tok"][u])])
        want_tiles = 0 if last < 0 else last // BN + 1
        assert t["n_tiles"][u] == want_tiles
    assert np.all(covered == 1)


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
@pytest.mark.parametrize("case", CASES + [(W.chunked().q_lens, W.chunked().k_lens, 32, 8, 128, 152)] +
                         random_cases(24) + [([512000], [9000000], 1, 1, 64, 1024)])
def test_group_major_list_assignment(case):
    lq, lk, Hq, Hkv, d, n_cta = case
    cu_q = np.concatenate([[0], np.cumsum(lq)]).astype(np.int32)
    cu_k = np.concatenate([[0], np.cumsum(lk)]).astype(np.int32)
    units, offs = pkg.opattn_schedule(cu_q, cu_k, Hq, Hkv, d, n_cta)
    n = len(units)
    if n == 0:
        return
    G = Hq // Hkv
    order = expected_order(lq, lk, Hkv, d, G)
    assert len(order) == n
    P = len(offs) - 1
    assert P == min(n_cta, n)
    assert offs[0] == 0 and offs[-1] == n and np.all(np.diff(offs) >= 1)
    # replay the greedy list assignment and compare unit by unit
    import heapq
    heap = [(0, c) for c in range(P)]
    per_cta = [[] for _ in range(P)]
    for grp, n_tiles, s, h, t0 in order:
        load, c = heapq.heappop(heap)
        per_cta[c].append((s, h, t0, n_tiles))
        heapq.heappush(heap, (load + n_tiles + 1, c))
    t = unit_table(units)
    for c in range(P):
        got = [(int(t["seq"][i]), int(t["kvh"][i]), int(t["q_tok0"][i] - cu_q[t["seq"][i]]), int(t["n_tiles"][i]))
               for i in range(offs[c], offs[c + 1])]
        assert got == per_cta[c], f"CTA {c}"
    cost = units[:, 6].astype(np.int64) + 1
    loads = np.array([cost[offs[c]:offs[c + 1]].sum() for c in range(P)])
    assert loads.max() <= cost.sum() / P + cost.max() + 1e-9


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
    units = np.zeros((2, 8), dtype=np.int32)
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
