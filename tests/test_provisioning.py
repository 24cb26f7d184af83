"""Queueing model (Eq. 2) and greedy provisioning (Algorithm 1), CPU only.

Erlang-C is pinned to closed forms (R = 1, 2), the textbook factorial sum in
exact rational arithmetic, the stationary distribution of the M/M/R
birth-death chain, and a discrete-event simulation.  The greedy plan search
is checked against the exhaustive search on seeded random operator graphs,
and on hand-built cases that force scaling up, scaling down and an
unreachable SLO.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

from paper_2608_13499_gb300 import provisioning as V


# ------------------------------------------------------------ Erlang-C pins

@pytest.mark.parametrize("rho", [0.0, 0.1, 0.5, 0.9, 0.999])
def test_erlang_c_single_and_two_servers(rho):
    assert abs(V.erlang_c(1, rho) - rho) < 1e-15              # M/M/1: P(wait) = rho
    assert abs(V.erlang_c(2, rho) - 2 * rho * rho / (1 + rho)) < 1e-15


def erlang_c_factorial_sum(R, a):
    """Textbook form with exact rationals: (a^R/R! R/(R-a)) / (sum_{k<R} a^k/k! + a^R/R! R/(R-a))."""
    a = Fraction(a)
    top = a ** R / math.factorial(R) * Fraction(R) / (R - a)
    return top / (sum(a ** k / math.factorial(k) for k in range(R)) + top)


@pytest.mark.parametrize("R,a", [(3, Fraction(5, 2)), (8, Fraction(6)), (25, Fraction(47, 2)), (64, Fraction(40)),
                                 (150, Fraction(149))])
def test_erlang_c_matches_factorial_sum(R, a):
    want = float(erlang_c_factorial_sum(R, a))
    assert abs(V.erlang_c(R, float(a) / R) - want) <= 1e-12 * max(want, 1e-300)


@pytest.mark.parametrize("lam,mu,R", [(3.2, 1.0, 4), (0.5, 2.0, 1), (17.0, 0.75, 25), (9.9, 1.0, 10)])
def test_waiting_time_matches_birth_death_chain(lam, mu, R):
    # stationary distribution pi_n proportional to prod_k lam / (min(k, R) mu), truncated far out
    N = 20000
    logw = np.zeros(N)
    for n in range(1, N):
        logw[n] = logw[n - 1] + math.log(lam / (min(n, R) * mu))
    pi = np.exp(logw - logw.max())
    pi /= pi.sum()
    p_wait = pi[R:].sum()
    wq = (np.arange(N - R) * pi[R:]).sum() / lam             # Little's law on the queue
    assert abs(V.erlang_c(R, lam / (R * mu)) - p_wait) < 1e-9
    assert abs(V.waiting_time(lam, R, mu) - wq) < 1e-9 * max(1.0, wq)


def test_waiting_time_matches_simulation():
    lam, mu, R = 3.2, 1.0, 4
    sim = V.simulate_mmr(lam, mu, R, 400000, seed=1)
    assert abs(sim / V.waiting_time(lam, R, mu) - 1.0) < 0.05


def test_stability_edges():
    assert V.waiting_time(2.0, 2, 1.0) == math.inf          # rho = 1
    assert V.waiting_time(5.0, 2, 1.0) == math.inf
    assert V.waiting_time(0.0, 3, 1.0) == 0.0
    assert V.erlang_c(3, 1.0) == 1.0
    assert V.min_stable_replicas(4.0, 1.0) == 5             # ceil would give rho = 1
    assert V.min_stable_replicas(4.5, 1.0) == 5
    assert V.min_stable_replicas(0.2, 1.0) == 1
    # more replicas never wait longer; a busier queue never waits less
    assert all(V.erlang_c(r + 1, 7.0 / (r + 1)) < V.erlang_c(r, 7.0 / r) for r in range(8, 20))
    assert all(V.erlang_c(6, x) < V.erlang_c(6, x + 0.05) for x in np.linspace(0.05, 0.9, 18))


# ------------------------------------------------------------ the DAG

def op(name, t, b_max=8, shards=(1,), visits=1, comm=0.0, deps=()):
    return V.Operator(name, t, b_max, shards, visits, comm, deps)


def test_service_rate_follows_the_appendix():
    o = op("attn", lambda b, p: 0.002 + 0.001 * b, visits=32)
    assert abs(o.mu(1, 1) - 1.0 / (0.003 * 32)) < 1e-12     # mu = 1 / (op_latency * num_layers)
    assert abs(o.mu(4, 1) - 4.0 / (0.006 * 32)) < 1e-12


def test_critical_path_and_cycles():
    ops = [op("a", None), op("b", None, deps=("a",)), op("c", None, deps=("a",)), op("d", None, deps=("b", "c"))]
    lat, path = V.critical_path(ops, {"a": 1.0, "b": 5.0, "c": 2.0, "d": 0.5})
    assert lat == 6.5 and path == ["a", "b", "d"]
    lat, path = V.critical_path(ops, {"a": 1.0, "b": 1.0, "c": 2.0, "d": 0.5})
    assert lat == 3.5 and path == ["a", "c", "d"]
    with pytest.raises(ValueError):
        V.topological_order([op("x", None, deps=("y",)), op("y", None, deps=("x",))])
    with pytest.raises(ValueError):
        V.topological_order([op("x", None, deps=("z",))])


def test_chain_latency_is_eq1_sum():
    t = [lambda b, p: 0.001 + 0.0004 * b, lambda b, p: 0.003 + 0.002 * b, lambda b, p: 0.0005 * b]
    ops = [op(f"o{i}", t[i], comm=1e-4 * i, deps=((f"o{i-1}",) if i else ())) for i in range(3)]
    prov = V.Provisioner(ops, qps=300.0, slo=1.0)
    cfg = {"o0": V.OpConfig(1, 2, 1), "o1": V.OpConfig(3, 4, 1), "o2": V.OpConfig(1, 1, 1)}
    lat, path, s = prov.evaluate(cfg)
    want = 0.0
    for i, o in enumerate(ops):
        c = cfg[o.name]
        mu = c.b / t[i](c.b, 1)
        want += V.waiting_time(300.0, c.r, mu) + 1.0 / mu + o.comm
    assert abs(lat - want) < 1e-15 and path == ["o0", "o1", "o2"]


# ------------------------------------------------------------ Algorithm 1

def random_graph(rng, n):
    ops = []
    for i in range(n):
        t0, c, alpha, eff = rng.uniform(0.5e-3, 5e-3), rng.uniform(0.05e-3, 1e-3), rng.uniform(0.6, 1.0), \
            rng.uniform(0.6, 0.95)

        def lat(b, p, t0=t0, c=c, alpha=alpha, eff=eff):
            return (t0 + c * b ** alpha) / (1.0 if p == 1 else p * eff)
        deps = () if i == 0 else ((f"op{i-1}",) if rng.integers(0, 2) else (f"op{rng.integers(0, i)}",))
        ops.append(op(f"op{i}", lat, b_max=int(rng.integers(4, 13)), shards=(1, 2, 4),
                      visits=int(rng.integers(1, 4)), deps=deps))
    return ops


def instances(n, seed=0):
    rng = np.random.default_rng(seed)
    for _ in range(n):
        ops = random_graph(rng, int(rng.integers(2, 4)))
        qps = rng.uniform(200, 3000)
        base = V.Provisioner(ops, qps, 1.0)
        t0 = base.evaluate({o.name: base._initial(o) for o in base.ops})[0]
        yield ops, qps, t0 * rng.uniform(0.6, 2.0)


def test_greedy_cost_close_to_exhaustive_search():
    ratios = []
    for ops, qps, slo in instances(16):
        bf = V.brute_force_plan(ops, qps, slo)
        g = V.provision(ops, qps, slo)
        if bf is None:
            continue
        assert g.meets(slo), (g.latency, slo)
        assert g.cost >= bf.cost                              # the exhaustive search is optimal
        ratios.append(g.cost / bf.cost)
        for name, c in g.configs.items():                     # every queue is stable
            o = next(o for o in ops if o.name == name)
            assert qps < c.r * o.mu(c.b, c.p)
        assert abs(V.Provisioner(ops, qps, slo).evaluate(g.configs)[0] - g.latency) < 1e-15
    assert len(ratios) >= 12
    assert np.mean(ratios) <= 1.08                            # the paper: within 8% of the oracle


def test_scaling_up_reaches_a_tight_slo():
    t = lambda b, p: (0.004 + 0.001 * b) / (1.0 if p == 1 else 0.8 * p)
    ops = [op("a", t, b_max=8, shards=(1, 2)), op("b", lambda b, p: 0.001 * b, deps=("a",))]
    prov = V.Provisioner(ops, qps=900.0, slo=1.0)
    init = {o.name: prov._initial(o) for o in prov.ops}
    t_init = prov.evaluate(init)[0]
    slo = 0.8 * t_init
    plan = V.provision(ops, 900.0, slo)
    assert plan.meets(slo)
    assert any(s[0] == "up" for s in plan.steps)
    assert plan.cost > V.Provisioner.cost(init)


def test_scaling_down_reclaims_under_a_loose_slo():
    t = lambda b, p: 0.002 + 0.0005 * b
    ops = [op("a", t, b_max=16), op("b", lambda b, p: 0.003 + 0.0002 * b, b_max=16, deps=("a",))]
    prov = V.Provisioner(ops, qps=2000.0, slo=1.0)
    init = {o.name: prov._initial(o) for o in prov.ops}
    plan = V.provision(ops, 2000.0, 10.0 * prov.evaluate(init)[0])
    assert any(s[0] == "down" for s in plan.steps)
    assert plan.cost < V.Provisioner.cost(init)
    bf = V.brute_force_plan(ops, 2000.0, 10.0 * prov.evaluate(init)[0])
    assert plan.cost == bf.cost


def test_unreachable_slo_terminates_without_meeting_it():
    ops = [op("a", lambda b, p: 0.01 + 0.001 * b)]
    # the service time per request T(b)/b is at least 2.25 ms (b = 8)
    plan = V.provision(ops, 100.0, 0.002)
    assert not plan.meets(0.002)
    assert len(plan.steps) < 200
    assert V.brute_force_plan(ops, 100.0, 0.002) is None


@pytest.mark.parametrize("mode", ["bottleneck", "noncritical"])
def test_both_downscale_readings_meet_the_slo(mode):
    for ops, qps, slo in instances(6, seed=3):
        plan = V.provision(ops, qps, slo, downscale=mode)
        if V.brute_force_plan(ops, qps, slo) is not None:
            assert plan.meets(slo)


def test_latency_from_profile():
    from paper_2608_13499_gb300 import profiler as P
    pts = P.sample_points(10, np.random.default_rng(0), [(1, 32), (128, 8192)])
    prof = P.PiecewiseProfile(pts, 1e-4 * pts[:, 0] * pts[:, 1] ** 1.5)   # ms
    T = V.latency_from_profile(prof, 2048, tp_efficiency=0.5)
    assert abs(T(4, 1) - 1e-7 * 4 * 2048 ** 1.5) < 1e-12
    assert abs(T(4, 2) - T(4, 1)) < 1e-15                                   # 2 shards at 50% efficiency
