"""Operator profile of the prefill-attention operator.

OpScale provisions each operator from a profile of its latency over batch
size B, prompt length L and SM share S (§4.1, "Operator Profiling Space"),
built by sparse sampling: random points of the (B, L) space are measured and
unsampled points are estimated by non-parametric piecewise interpolation
(§4.2).  Operators that are structurally identical (the same attention in
every layer, or in two models with the same head geometry) share one profile
(§4.2, structural equivalence).  This module does that for libopattn:

* ``PiecewiseProfile``: piecewise-linear interpolation of log T over the log
  of each coordinate ((B, L) or (B, L, S)) on a Delaunay triangulation of the
  sampled points.  In log space the operator's O(L^2 B) cost (§2.1) is close
  to linear, so few samples suffice.  The corners of the sampled box are
  always in the sample, so every query inside the box is inside the
  triangulation.
* ``sample_points``: random points (a Latin hypercube in log space) plus
  the box corners.
* ``ProfileStore``: profiles keyed by the operator's structure, so that each
  distinct attention shape of a model is measured once.
* ``measure_ms``: CUDA-event time of one launch (``opattn_plan_run``) for a
  batch of B prompts of L tokens, with the persistent grid optionally capped
  at ``max_ctas`` CTAs.  The kernel keeps one CTA per SM, so the cap is the
  operator's SM budget S (the paper's S_v, §3.1).
* ``sm_budget_curve``: latency against SM share for a workload.
* ``colocate``: two operators (prefill and decode) running at once on
  disjoint SM budgets, against time slicing the whole GPU between them.
* ``profile_accuracy``: relative error of an interpolated profile on
  held-out random points.  The paper's operator profiles reach 7% mean and
  15% P90 relative error (§5, "Profiling-driven Model Accuracy").

``python -m paper_2608_13499_gb300.profiler --out FILE`` on a GPU writes a
markdown report of the studies.
"""
from __future__ import annotations

import argparse
import json
import math
import statistics
from dataclasses import asdict, dataclass

import numpy as np


class PiecewiseProfile:
    """Piecewise-linear interpolation of log T over log-coordinates.

    ``coords`` is an (n, k) array of positive sample coordinates (k = 2 for
    (B, L), 3 for (B, L, S)), ``times_ms`` the n measured latencies.
    """

    def __init__(self, coords, times_ms):
        from scipy.interpolate import LinearNDInterpolator
        x = np.asarray(coords, dtype=np.float64)
        t = np.asarray(times_ms, dtype=np.float64)
        if x.ndim != 2 or len(x) != len(t):
            raise ValueError("coords must be (n, k) with one time per row")
        if len(t) < x.shape[1] + 1:
            raise ValueError(f"need at least {x.shape[1] + 1} samples in {x.shape[1]} dimensions")
        if np.any(x <= 0) or np.any(t <= 0) or not np.all(np.isfinite(t)):
            raise ValueError("coordinates and times must be positive")
        self.coords = x
        self.times_ms = t
        self._x = np.log(x)
        self._logt = np.log(t)
        self._interp = LinearNDInterpolator(self._x, self._logt)

    @property
    def dims(self) -> int:
        return self.coords.shape[1]

    def predict(self, coords) -> np.ndarray:
        """Estimated times (ms) at an (m, k) array of points.

        Outside the convex hull of the samples the nearest sample (in log
        coordinates) answers, so the profile never extrapolates.
        """
        x = np.log(np.atleast_2d(np.asarray(coords, dtype=np.float64)))
        if x.shape[1] != self.dims:
            raise ValueError(f"points have {x.shape[1]} coordinates, the profile {self.dims}")
        out = np.asarray(self._interp(x), dtype=np.float64).reshape(len(x))
        miss = ~np.isfinite(out)
        if miss.any():
            d = ((x[miss, None, :] - self._x[None, :, :]) ** 2).sum(-1)
            out[miss] = self._logt[d.argmin(axis=1)]
        return np.exp(out)

    def to_dict(self) -> dict:
        return {"coords": self.coords.tolist(), "times_ms": self.times_ms.tolist()}

    @classmethod
    def from_dict(cls, d: dict) -> "PiecewiseProfile":
        return cls(d["coords"], d["times_ms"])


def sample_points(n: int, rng, ranges, integer=None, corners: bool = True, stratified: bool = True) -> np.ndarray:
    """(n [+ 2^k], k) random points, log-uniform in each range of ``ranges``.

    ``stratified`` draws a Latin hypercube in log space (each coordinate's
    log range cut into n equal strata, one point per stratum, strata paired
    at random across coordinates), which avoids the long thin triangles that
    clustered plain random points leave.  ``integer[i]`` rounds coordinate i
    (batch size, length); ``corners`` prepends the 2^k corners of the box.
    """
    k = len(ranges)
    integer = [True] * k if integer is None else list(integer)
    cols = []
    for (lo, hi), is_int in zip(ranges, integer):
        u = (rng.permutation(n) + rng.uniform(0.0, 1.0, n)) / n if stratified else rng.uniform(0.0, 1.0, n)
        c = np.exp(math.log(lo) + u * (math.log(hi) - math.log(lo)))
        if is_int:
            c = np.rint(c)
        cols.append(np.clip(c, lo, hi))
    pts = np.column_stack(cols) if n else np.zeros((0, k))
    if corners:
        box = np.array([[ranges[i][(m >> i) & 1] for i in range(k)] for m in range(1 << k)], dtype=np.float64)
        pts = np.concatenate([box, pts])
    return pts


def relative_errors(predicted, measured) -> dict:
    p, m = np.asarray(predicted, dtype=np.float64), np.asarray(measured, dtype=np.float64)
    e = np.abs(p - m) / m
    return {"mean": float(e.mean()), "p90": float(np.percentile(e, 90)), "max": float(e.max()), "n": int(len(e))}


# ------------------------------------------------------- structural equivalence

@dataclass(frozen=True)
class OperatorKey:
    """What decides an operator's latency: its kernel, shape parameters and dtype.

    Layers (and models) whose operator has the same key run the same kernel
    on the same shapes, so one profile serves them all.
    """
    op: str
    shape: tuple
    dtype: str = "bf16"

    def name(self) -> str:
        return f"{self.op}{list(self.shape)}/{self.dtype}"


def attention_key(Hq: int, Hkv: int, d: int) -> OperatorKey:
    """The prefill-attention operator with Hq query heads, Hkv kv heads, head size d."""
    return OperatorKey("opattn_prefill", (int(Hq), int(Hkv), int(d)))


def decode_key(Hq: int, Hkv: int, d: int) -> OperatorKey:
    """The decode-attention operator (one query token per request over its cached keys)."""
    return OperatorKey("opattn_decode", (int(Hq), int(Hkv), int(d)))


def gemm_key(k_in: int, n_out: int) -> OperatorKey:
    """A token-wise projection: [tokens, k_in] x [k_in, n_out]."""
    return OperatorKey("gemm", (int(k_in), int(n_out)))


class ProfileStore:
    """Profiles by operator key; ``get`` profiles a key only the first time."""

    def __init__(self):
        self._profiles: dict = {}
        self.measured: list = []     # keys in the order they were profiled

    def __contains__(self, key: OperatorKey) -> bool:
        return key in self._profiles

    def __len__(self) -> int:
        return len(self._profiles)

    def __getitem__(self, key: OperatorKey) -> PiecewiseProfile:
        return self._profiles[key]

    def get(self, key: OperatorKey, profile_fn) -> PiecewiseProfile:
        if key not in self._profiles:
            self._profiles[key] = profile_fn(key)
            self.measured.append(key)
        return self._profiles[key]

    def profiles_for(self, layer_keys, profile_fn) -> list:
        """One profile per layer, measuring each distinct key once."""
        return [self.get(k, profile_fn) for k in layer_keys]

    def save(self, path: str) -> None:
        blob = [{"key": asdict(k), "profile": p.to_dict()} for k, p in self._profiles.items()]
        with open(path, "w") as f:
            json.dump(blob, f)

    @classmethod
    def load(cls, path: str) -> "ProfileStore":
        s = cls()
        with open(path) as f:
            for e in json.load(f):
                k = e["key"]
                key = OperatorKey(k["op"], tuple(k["shape"]), k["dtype"])
                s._profiles[key] = PiecewiseProfile.from_dict(e["profile"])
        return s


# ---------------------------------------------------------------- GPU side

class _Buffers:
    """Device inputs sized for the largest point; every point uses a prefix.

    ``max_queries`` query rows (default: as many as keys) and ``max_keys`` key rows.
    """

    def __init__(self, max_keys: int, Hq: int, Hkv: int, d: int, device="cuda", max_queries: int = 0):
        import torch

        from . import workloads as W
        self.Hq, self.Hkv, self.d = Hq, Hkv, d
        n, nq = max_keys, max_queries or max_keys
        self.q = W.normal_bf16(0, W.STREAM_Q, nq * Hq * d, device).view(nq, Hq, d)
        self.k = W.normal_bf16(0, W.STREAM_K, n * Hkv * d, device).view(n, Hkv, d)
        self.v = W.normal_bf16(0, W.STREAM_V, n * Hkv * d, device).view(n, Hkv, d)
        self.o = torch.empty((nq, Hq, d), dtype=torch.bfloat16, device=device)
        self.lse = torch.empty((nq, Hq), dtype=torch.float32, device=device)


def time_callable_ms(fn, reps: int, warm_ms: float = 25.0, min_ms: float = 2.0) -> float:
    """Median per-call CUDA-event time (ms) of ``fn`` launching work on the current stream.

    ``fn`` first runs back to back for ``warm_ms`` so the clocks leave their
    idle state.  Each of the ``reps`` samples then times ``inner`` back-to-back
    calls between two events (``inner`` chosen so a sample spans at least
    ``min_ms``), so the host's launch gap before a single short launch is not
    counted.
    """
    import torch
    stream = torch.cuda.current_stream()

    def sample(inner):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(inner):
            fn()
        b.record(stream)
        b.synchronize()
        return a.elapsed_time(b) / inner

    first = sample(1)
    inner = max(1, min(256, int(math.ceil(min_ms / max(first, 1e-3)))))
    warm = 0.0
    while warm < warm_ms:
        warm += sample(inner) * inner
    return statistics.median(sample(inner) for _ in range(reps))


def _time_plan_ms(plan, q, k, v, o, lse, scale, reps: int) -> float:
    import torch
    stream = torch.cuda.current_stream()
    return time_callable_ms(lambda: plan.run(q, k, v, o, lse, scale, stream), reps)


def n_sms() -> int:
    import torch
    return torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count


def ctas_for_share(share: float, sms: int) -> int:
    """SM count for an SM share in (0, 1]: round(share * sms), at least 1."""
    return max(1, min(sms, int(round(share * sms))))


def measure_ms(buf, B: int, L: int, max_ctas: int = 0, reps: int = 5) -> float:
    """Median time (ms) of one launch for B prompts of L tokens each (q_len = kv_len = L)."""
    import paper_2608_13499_gb300 as pkg
    cu = np.arange(B + 1, dtype=np.int32) * np.int32(L)
    with pkg.Plan(cu, cu, buf.Hq, buf.Hkv, buf.d, max_ctas=max_ctas) as plan:
        return _time_plan_ms(plan, buf.q, buf.k, buf.v, buf.o, buf.lse, buf.d ** -0.5, reps)


def measure_decode_ms(buf, B: int, L: int, max_ctas: int = 0, reps: int = 5) -> float:
    """Median time (ms) of one decode launch: B requests, one query token each, L cached keys each."""
    import paper_2608_13499_gb300 as pkg
    cu_q = np.arange(B + 1, dtype=np.int32)
    cu_k = cu_q * np.int32(L)
    with pkg.Plan(cu_q, cu_k, buf.Hq, buf.Hkv, buf.d, max_ctas=max_ctas, decode=True) as plan:
        return _time_plan_ms(plan, buf.q, buf.k, buf.v, buf.o, buf.lse, buf.d ** -0.5, reps)


def sm_budget_curve(w, ctas, reps: int = 5, device="cuda", decode: bool = False):
    """[(n_ctas, ms)] for workload w with the persistent grid capped at each budget."""
    import torch

    import paper_2608_13499_gb300 as pkg

    from . import workloads as W
    q, k, v = W.make_inputs(w, device)
    o = torch.empty((w.total_q, w.Hq, w.d), dtype=torch.bfloat16, device=device)
    lse = torch.empty((w.total_q, w.Hq), dtype=torch.float32, device=device)
    out = []
    for n in ctas:
        with pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, max_ctas=n, decode=decode) as plan:
            out.append((plan.n_ctas, _time_plan_ms(plan, q, k, v, o, lse, w.scale, reps)))
    return out


def colocate(w_a, w_b, ctas_a: int, ctas_b: int, decode_a: bool = False, decode_b: bool = True,
             span_ms: float = 20.0, reps: int = 3, device="cuda") -> dict:
    """Two operators sharing the GPU spatially (§2.1, "Sensitivity to SM Core Allocation").

    Operator A (workload ``w_a``) runs with its persistent grid capped at
    ``ctas_a`` CTAs on one stream, operator B at ``ctas_b`` on another; with
    ``ctas_a + ctas_b`` at most the SM count and one CTA per SM, both grids
    are resident at once on disjoint SMs, and neither kernel waits on the
    other.  Each stream gets about ``span_ms`` of launches (counted from the
    operator's time alone at its budget), all queued behind one event so
    that they start together.  Returns the per-launch times alone (at the
    budget and at the full GPU) and co-located, each operator's interference
    factor I = co-located / alone at the same SM allocation (§4.4), and the
    co-located makespan against running the same launches one operator after
    the other on the whole GPU (time slicing).
    """
    import torch

    import paper_2608_13499_gb300 as pkg

    from . import workloads as W
    sms = n_sms()
    if ctas_a + ctas_b > sms:
        raise ValueError(f"budgets {ctas_a} + {ctas_b} exceed the {sms} SMs")

    def operator(w, dec, n):
        q, k, v = W.make_inputs(w, device)
        o = torch.empty((w.total_q, w.Hq, w.d), dtype=torch.bfloat16, device=device)
        lse = torch.empty((w.total_q, w.Hq), dtype=torch.float32, device=device)
        plan = pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, max_ctas=n, decode=dec)
        full = pkg.Plan(w.cu_q, w.cu_k, w.Hq, w.Hkv, w.d, decode=dec)
        return plan, full, (q, k, v, o, lse, w.scale)

    plan_a, full_a, args_a = operator(w_a, decode_a, ctas_a)
    plan_b, full_b, args_b = operator(w_b, decode_b, ctas_b)
    try:
        alone_a, alone_b = _time_plan_ms(plan_a, *args_a, reps), _time_plan_ms(plan_b, *args_b, reps)
        full_ms_a, full_ms_b = _time_plan_ms(full_a, *args_a, reps), _time_plan_ms(full_b, *args_b, reps)
        n_a = max(1, int(math.ceil(span_ms / alone_a)))
        n_b = max(1, int(math.ceil(span_ms / alone_b)))
        main = torch.cuda.current_stream()
        s_a, s_b = torch.cuda.Stream(), torch.cuda.Stream()
        samples = []
        for _ in range(reps):
            start = torch.cuda.Event(enable_timing=True)
            end_a, end_b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda._sleep(10_000_000)  # a few ms, so that every launch below is queued before the start
            start.record(main)
            s_a.wait_event(start)
            s_b.wait_event(start)
            for _ in range(n_a):
                plan_a.run(*args_a, s_a)
            end_a.record(s_a)
            for _ in range(n_b):
                plan_b.run(*args_b, s_b)
            end_b.record(s_b)
            end_a.synchronize()
            end_b.synchronize()
            samples.append((start.elapsed_time(end_a), start.elapsed_time(end_b)))
        main.wait_stream(s_a)
        main.wait_stream(s_b)
        t_a = statistics.median(a for a, _ in samples)
        t_b = statistics.median(b for _, b in samples)
        makespan = statistics.median(max(a, b) for a, b in samples)
        sliced = n_a * full_ms_a + n_b * full_ms_b
        return {"ctas": (ctas_a, ctas_b), "launches": (n_a, n_b), "alone_ms": (alone_a, alone_b),
                "full_gpu_ms": (full_ms_a, full_ms_b), "colocated_ms": (t_a / n_a, t_b / n_b),
                "interference": (t_a / n_a / alone_a, t_b / n_b / alone_b),
                "makespan_ms": makespan, "time_sliced_ms": sliced, "speedup": sliced / makespan}
    finally:
        for p in (plan_a, full_a, plan_b, full_b):
            p.close()


class GemmOperator:
    """Times a bf16 token-wise projection (library matmul) for B prompts of L tokens."""

    def __init__(self, k_in: int, n_out: int, max_tokens: int, device="cuda"):
        import torch
        g = torch.Generator(device=device)
        g.manual_seed(0)
        self.x = torch.randn((max_tokens, k_in), generator=g, device=device, dtype=torch.bfloat16)
        self.w = torch.randn((k_in, n_out), generator=g, device=device, dtype=torch.bfloat16) * k_in ** -0.5
        self.y = torch.empty((max_tokens, n_out), device=device, dtype=torch.bfloat16)

    def measure(self, B: int, L: int, reps: int = 5) -> float:
        import torch
        m = B * L
        return time_callable_ms(lambda: torch.matmul(self.x[:m], self.w, out=self.y[:m]), reps)


def profile_operator(measure, n_train: int, rng, b_range=(1, 32), l_range=(128, 8192)) -> PiecewiseProfile:
    """Sparse-sampling profile over (B, L) of any ``measure(B, L) -> ms``."""
    pts = sample_points(n_train, rng, [b_range, l_range])
    return PiecewiseProfile(pts, [measure(int(b), int(x)) for b, x in pts])


def llama3_8b_layer_keys():
    """The operators of one Llama-3-8B decoder layer that the provisioning study uses."""
    return {"qkv_proj": gemm_key(4096, 6144), "attention": attention_key(32, 8, 128),
            "o_proj": gemm_key(4096, 4096), "gate_up_proj": gemm_key(4096, 28672),
            "down_proj": gemm_key(14336, 4096)}


def build_store(n_train: int, seed: int = 0, b_range=(1, 32), l_range=(128, 8192), reps: int = 5) -> ProfileStore:
    """Profiles of every distinct operator of Llama-3-8B's 32 layers (each measured once)."""
    import torch
    rng = np.random.default_rng(seed)
    max_tokens = int(b_range[1] * l_range[1])
    store = ProfileStore()

    def profile(key):
        if key.op == "opattn_prefill":
            buf = _Buffers(max_tokens, *key.shape)
            fn = lambda B, L: measure_ms(buf, B, L, reps=reps)
        else:
            g = GemmOperator(key.shape[0], key.shape[1], max_tokens)
            fn = lambda B, L: g.measure(B, L, reps)
        prof = profile_operator(fn, n_train, rng, b_range, l_range)
        torch.cuda.empty_cache()
        return prof

    layers = [k for _ in range(32) for k in llama3_8b_layer_keys().values()]
    store.profiles_for(layers, profile)
    return store


def profile_accuracy(n_train: int, n_test: int, seed: int = 0, key: OperatorKey = attention_key(32, 8, 128),
                     b_range=(1, 32), l_range=(128, 8192), s_range=None, reps: int = 5):
    """Fit a profile on n_train random points plus the box corners; error on n_test others.

    With ``s_range`` (SM shares, e.g. (1/16, 1)) the profile is over (B, L, S).  A
    ``decode_key`` profiles the decode operator: B requests of one query token
    over L cached keys each.
    """
    rng = np.random.default_rng(seed)
    ranges = [b_range, l_range] + ([s_range] if s_range else [])
    integer = [True, True] + ([False] if s_range else [])
    train = sample_points(n_train, rng, ranges, integer)
    test = sample_points(n_test, rng, ranges, integer, corners=False, stratified=False)
    decode = key.op == "opattn_decode"
    buf = _Buffers(int(b_range[1] * l_range[1]), *key.shape, max_queries=int(b_range[1]) if decode else 0)
    measure = measure_decode_ms if decode else measure_ms
    sms = n_sms()

    def run(p):
        ctas = ctas_for_share(p[2], sms) if s_range else 0
        return measure(buf, int(p[0]), int(p[1]), ctas, reps)

    t_train = np.array([run(p) for p in train])
    t_test = np.array([run(p) for p in test])
    t_again = np.array([run(p) for p in test])
    prof = PiecewiseProfile(train, t_train)
    pred = prof.predict(test)
    return {"profile": prof, "test": test, "measured": t_test, "predicted": pred,
            "errors": relative_errors(pred, t_test), "noise": relative_errors(t_again, t_test),
            "remeasured": t_again}


def _accuracy_section(title, acc, n_train, k) -> list:
    e = acc["errors"]
    lines = [f"## {title}", "",
             f"{len(acc['profile'].coords)} sampled points ({1 << k} box corners + {n_train} random points, "
             f"a Latin hypercube in log space), {e['n']} held-out log-uniform random points.", "",
             "| relative error of the interpolated latency | value |", "|---|---|",
             f"| mean | {100 * e['mean']:.1f}% |", f"| P90 | {100 * e['p90']:.1f}% |",
             f"| max | {100 * e['max']:.1f}% |", "",
             f"Measurement noise (the held-out points timed twice): {100 * acc['noise']['mean']:.1f}% mean, "
             f"{100 * acc['noise']['p90']:.1f}% P90.", "",
             "| " + " | ".join(["B", "L", "S"][:k]) + " | measured (ms) | predicted (ms) |",
             "|" + "---|" * (k + 2)]
    for p, t, q in list(zip(acc["test"], acc["measured"], acc["predicted"]))[:10]:
        cells = [str(int(p[0])), str(int(p[1]))] + ([f"{p[2]:.3f}"] if k == 3 else [])
        lines.append("| " + " | ".join(cells) + f" | {t:.4f} | {q:.4f} |")
    return lines + [""]


def _report(args) -> str:
    import torch

    from . import workloads as W
    sms = n_sms()
    lines = ["# Operator profiles of opattn_prefill and opattn_decode: sparse sampling, piecewise "
             "interpolation, SM budget", "",
             f"Command: `python -m paper_2608_13499_gb300.profiler --train {args.train} --test {args.test} "
             f"--train3 {args.train3} --test3 {args.test3} --seed {args.seed} --reps {args.reps} --out <file>"
             f"{' --dump <file>' if args.dump else ''}` "
             f"on one {torch.cuda.get_device_name(0)} ({sms} SMs).", "",
             "Each point is the median of "
             f"{args.reps} CUDA-event samples after 25 ms of back-to-back warm-up launches; a sample times "
             "enough back-to-back launches to span 2 ms and divides.  Inputs N(0, 1) bf16.  The paper's "
             "operator profiles: 7% mean and 15% P90 relative error.", "",
             "Prefill operator: Llama-3-8B attention heads (Hq 32, Hkv 8, d 128), B prompts of L tokens each, "
             "B in [1, 32], L in [128, 8192].", ""]
    acc2 = profile_accuracy(args.train, args.test, args.seed, reps=args.reps)
    lines += _accuracy_section("Prefill profile over (B, L) at the full GPU", acc2, args.train, 2)
    acc3 = profile_accuracy(args.train3, args.test3, args.seed + 1, s_range=(1.0 / 16, 1.0), reps=args.reps)
    lines += _accuracy_section("Prefill profile over (B, L, S), SM share S in [1/16, 1]", acc3, args.train3, 3)
    lines += ["Decode operator: Llama-3-70B attention heads (Hq 64, Hkv 8, d 128), B requests of one query "
              "token over L cached keys each, B in [1, 256], L in [256, 32768].", ""]
    accd = profile_accuracy(args.train, args.test, args.seed + 2, key=decode_key(64, 8, 128), b_range=(1, 256),
                            l_range=(256, 32768), reps=args.reps)
    lines += _accuracy_section("Decode profile over (B, L) at the full GPU", accd, args.train, 2)
    if args.dump:
        blob = {name: {"train": a["profile"].to_dict(), "test": a["test"].tolist(),
                       "measured": a["measured"].tolist(), "remeasured": a["remeasured"].tolist()}
                for name, a in (("BL", acc2), ("BLS", acc3), ("decode_BL", accd))}
        with open(args.dump, "w") as f:
            json.dump(blob, f)
    shares = (0.125, 0.25, 0.5, 0.75, 1.0)
    budgets = [ctas_for_share(f, sms) for f in shares]
    lines += [f"## Latency against SM budget (persistent grid capped at n CTAs, one CTA per SM)", "",
              "Time relative to the full GPU in parentheses; perfect scaling would be 1/share.", "",
              "| workload | " + " | ".join(f"{b} SMs ({100 * b / sms:.0f}%)" for b in budgets) + " |",
              "|---|" + "---|" * len(budgets)]
    rows = [(W.STANDARD[n](), False) for n in ("llama3_8b", "llama3_70b", "bursty", "chunked")]
    rows += [(W.DECODE[n](), True) for n in ("decode_llama3_70b", "decode_llama3_8b")]
    for w, dec in rows:
        curve = sm_budget_curve(w, budgets, reps=args.reps, decode=dec)
        base = curve[-1][1]
        lines.append(f"| {w.name} | " + " | ".join(f"{ms:.3f} ms ({ms / base:.2f}x)" for _, ms in curve) + " |")
        torch.cuda.empty_cache()
    lines += [""] + _colocation_section(args.reps)
    return "\n".join(lines) + "\n"


def _colocation_section(reps: int) -> list:
    import torch

    from . import workloads as W
    sms = n_sms()
    wa, wb = W.STANDARD["llama3_70b"](), W.DECODE["decode_llama3_70b"]()
    lines = ["## Prefill and decode co-located on disjoint SM budgets", "",
             f"Prefill: {wa.name} (one Llama-3-70B layer's attention, compute-bound); decode: {wb.name} "
             "(HBM-bound).  Both run at once, each on its own stream with its persistent grid capped at its "
             "budget, for about 20 ms of launches each; 'time-sliced' runs the same launches one operator after "
             f"the other on all {sms} SMs.  I is the interference factor of §4.4: co-located over "
             f"alone at the same SM allocation.  Median of {reps} runs.", "",
             "| SMs prefill + decode | prefill ms: alone at budget / co-located (I) | decode ms: alone at budget / "
             "co-located (I) | makespan | time-sliced | speedup |", "|---|---|---|---|---|---|"]
    for frac_b in (0.125, 0.25, 0.375, 0.5, 0.625, 0.75):
        nb = ctas_for_share(frac_b, sms)
        r = colocate(wa, wb, sms - nb, nb, reps=reps)
        lines.append(f"| {sms - nb} + {nb} | {r['alone_ms'][0]:.3f} / {r['colocated_ms'][0]:.3f} "
                     f"({r['interference'][0]:.3f}) | {r['alone_ms'][1]:.3f} / {r['colocated_ms'][1]:.3f} "
                     f"({r['interference'][1]:.3f}) | {r['makespan_ms']:.1f} ms | "
                     f"{r['time_sliced_ms']:.1f} ms | {r['speedup']:.2f}x |")
        torch.cuda.empty_cache()
    lines += ["", f"Alone on all {sms} SMs: prefill {r['full_gpu_ms'][0]:.3f} ms, decode "
              f"{r['full_gpu_ms'][1]:.3f} ms per launch.", ""]
    half = sms // 2
    lines += [f"Other operator pairs, {half} + {sms - half} SMs (A + B):", "",
              "| A | B | A ms: alone at budget / co-located (I) | B ms: alone at budget / co-located (I) | "
              "speedup over time slicing |", "|---|---|---|---|---|"]
    pairs = [(W.STANDARD["llama3_70b"](), False, W.STANDARD["llama3_8b"](), False),
             (W.DECODE["decode_llama3_70b"](), True, W.DECODE["decode_llama3_8b"](), True)]
    for w1, d1, w2, d2 in pairs:
        r = colocate(w1, w2, half, sms - half, decode_a=d1, decode_b=d2, reps=reps)
        lines.append(f"| {w1.name} | {w2.name} | {r['alone_ms'][0]:.3f} / {r['colocated_ms'][0]:.3f} "
                     f"({r['interference'][0]:.3f}) | {r['alone_ms'][1]:.3f} / {r['colocated_ms'][1]:.3f} "
                     f"({r['interference'][1]:.3f}) | {r['speedup']:.2f}x |")
        torch.cuda.empty_cache()
    return lines + [""]


def main(argv=None):
    ap = argparse.ArgumentParser(description="profile opattn_prefill on the current GPU")
    ap.add_argument("--train", type=int, default=80)
    ap.add_argument("--test", type=int, default=40)
    ap.add_argument("--train3", type=int, default=160)
    ap.add_argument("--test3", type=int, default=40)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--reps", type=int, default=7)
    ap.add_argument("--out", default=None)
    ap.add_argument("--dump", default=None, help="write every measured point as JSON")
    ap.add_argument("--store", default=None,
                    help="only build the Llama-3-8B layer's operator profiles and save them here as JSON")
    ap.add_argument("--colocate", action="store_true",
                    help="only measure prefill and decode co-located on disjoint SM budgets")
    args = ap.parse_args(argv)
    from . import build
    build.build()
    if args.colocate:
        print("\n".join(_colocation_section(args.reps)))
        return
    if args.store:
        store = build_store(args.train, args.seed, reps=args.reps)
        store.save(args.store)
        print(f"{len(store)} operator profiles ({len(store.measured)} measured) -> {args.store}")
        return
    text = _report(args)
    if args.out:
        with open(args.out, "w") as f:
            f.write(text)
    print(text)


if __name__ == "__main__":
    main()
