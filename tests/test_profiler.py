"""Sparse-sampling operator profile (host side, no GPU).

The interpolation is checked against functions whose values are known
everywhere: a power law (affine in log space, so piecewise-linear
interpolation in log space must reproduce it exactly), an attention-like cost
with launch overhead, linear and quadratic terms (accuracy bound), and the
behaviour outside the sampled box (no extrapolation).
"""
import math

import numpy as np
import pytest

from paper_2608_13499_gb300 import profiler as P


def power_law(x):
    x = np.atleast_2d(x)
    return 3e-4 * x[:, 0] ** 1.0 * x[:, 1] ** 2.0 * (x[:, 2] ** -1.0 if x.shape[1] == 3 else 1.0)


def attention_like(x):
    """Launch overhead + per-token work + causal pairs, like a prefill kernel."""
    x = np.atleast_2d(x)
    B, L = x[:, 0], x[:, 1]
    return 0.008 + 2e-6 * B * L + 2.4e-8 * B * L * (L + 1) / 2


def test_sample_points_box_ranges_and_determinism():
    rng = np.random.default_rng(3)
    pts = P.sample_points(50, rng, [(1, 32), (128, 8192)])
    assert pts.shape == (54, 2)
    corners = {tuple(p) for p in pts[:4]}
    assert corners == {(1, 128), (1, 8192), (32, 128), (32, 8192)}
    assert np.all(pts[:, 0] >= 1) and np.all(pts[:, 0] <= 32)
    assert np.all(pts[:, 1] >= 128) and np.all(pts[:, 1] <= 8192)
    assert np.all(pts == np.rint(pts))
    again = P.sample_points(50, np.random.default_rng(3), [(1, 32), (128, 8192)])
    np.testing.assert_array_equal(pts, again)
    # log-uniform: about half of the lengths fall below the geometric midpoint 1024
    for stratified in (True, False):
        pts = P.sample_points(4000, rng, [(1, 32), (128, 8192)], corners=False, stratified=stratified)
        assert 0.45 < np.mean(pts[:, 1] < 1024) < 0.55
    # Latin hypercube: exactly one point in each of the n log strata of every coordinate
    lhs = P.sample_points(64, rng, [(0.5, 2.0), (10.0, 1e4)], [False, False], corners=False)
    for c, (lo, hi) in enumerate([(0.5, 2.0), (10.0, 1e4)]):
        strata = np.floor(64 * np.log(lhs[:, c] / lo) / math.log(hi / lo)).astype(int)
        assert sorted(strata) == list(range(64))
    three = P.sample_points(5, rng, [(1, 32), (128, 8192), (0.0625, 1.0)], [True, True, False])
    assert three.shape == (13, 3)
    assert np.any(three[8:, 2] != np.rint(three[8:, 2]))


def test_exact_at_the_samples():
    rng = np.random.default_rng(1)
    pts = P.sample_points(30, rng, [(1, 32), (128, 8192)])
    pts = np.unique(pts, axis=0)
    t = attention_like(pts)
    prof = P.PiecewiseProfile(pts, t)
    np.testing.assert_allclose(prof.predict(pts), t, rtol=1e-12)


@pytest.mark.parametrize("k", [2, 3])
def test_power_law_is_reproduced_everywhere(k):
    """T = c B L^2 / S is affine in log space: interpolation there is exact."""
    rng = np.random.default_rng(2)
    ranges = [(1, 32), (128, 8192), (0.0625, 1.0)][:k]
    integer = [True, True, False][:k]
    pts = np.unique(P.sample_points(20, rng, ranges, integer), axis=0)
    prof = P.PiecewiseProfile(pts, power_law(pts))
    q = P.sample_points(200, rng, ranges, [False] * k, corners=False, stratified=False)
    np.testing.assert_allclose(prof.predict(q), power_law(q), rtol=1e-9)


def test_a_dropped_quadratic_term_is_visible():
    """The interpolant follows the data, not a fixed model: it tracks L^2 growth."""
    rng = np.random.default_rng(4)
    pts = np.unique(P.sample_points(80, rng, [(1, 32), (128, 8192)]), axis=0)
    prof = P.PiecewiseProfile(pts, attention_like(pts))
    q = P.sample_points(400, rng, [(1, 32), (128, 8192)], corners=False, stratified=False)
    err = P.relative_errors(prof.predict(q), attention_like(q))
    # inside the paper's 7% mean / 15% P90 with room to spare for a smooth monotone cost
    assert err["mean"] < 0.03 and err["p90"] < 0.07
    # an interpolant of a cost without the quadratic term misses by a wide margin
    linear_only = lambda x: 0.008 + 2e-6 * x[:, 0] * x[:, 1]
    prof_lin = P.PiecewiseProfile(pts, linear_only(pts))
    assert P.relative_errors(prof_lin.predict(q), attention_like(q))["mean"] > 0.5


def test_no_extrapolation_outside_the_box():
    pts = np.array([[1, 128], [1, 8192], [32, 128], [32, 8192]], dtype=float)
    t = np.array([1.0, 2.0, 3.0, 4.0])
    prof = P.PiecewiseProfile(pts, t)
    got = prof.predict([[0.5, 100], [64, 20000], [1, 1e6]])
    np.testing.assert_allclose(got, [1.0, 4.0, 2.0])
    # inside: geometric mean of the corners at the centre of the log box
    centre = prof.predict([[math.sqrt(32), math.sqrt(128 * 8192)]])[0]
    assert min(t) < centre < max(t)


def test_relative_errors():
    e = P.relative_errors([1.1, 0.9, 2.0, 1.0], [1.0, 1.0, 1.0, 1.0])
    assert e["n"] == 4 and abs(e["mean"] - 0.3) < 1e-12 and e["max"] == 1.0
    assert abs(e["p90"] - np.percentile([0.1, 0.1, 1.0, 0.0], 90)) < 1e-12


@pytest.mark.parametrize("bad", [
    dict(coords=[[1, 1], [2, 2]], times=[1, 2]),                 # too few for 2-D
    dict(coords=[[1, 1], [2, 2], [0, 3]], times=[1, 2, 3]),      # non-positive coordinate
    dict(coords=[[1, 1], [2, 2], [1, 3]], times=[1, 2, -3]),     # non-positive time
    dict(coords=[[1, 1], [2, 2], [1, 3]], times=[1, 2]),         # length mismatch
])
def test_profile_rejects_bad_samples(bad):
    with pytest.raises(ValueError):
        P.PiecewiseProfile(bad["coords"], bad["times"])


def test_ctas_for_share():
    assert P.ctas_for_share(1.0, 152) == 152
    assert P.ctas_for_share(0.25, 152) == 38
    assert P.ctas_for_share(1e-6, 152) == 1
    assert P.ctas_for_share(2.0, 152) == 152


def test_structural_equivalence_profiles_each_shape_once(tmp_path):
    calls = []

    def fake_profile(key):
        calls.append(key)
        pts = np.array([[1, 128], [1, 8192], [32, 128], [32, 8192]], dtype=float)
        return P.PiecewiseProfile(pts, key.shape[0] * attention_like(pts))

    store = P.ProfileStore()
    llama3_70b = [P.attention_key(64, 8, 128)] * 80
    llama3_8b = [P.attention_key(32, 8, 128)] * 32
    llama31_8b = [P.attention_key(32, 8, 128)] * 32       # same attention as Llama-3-8B
    profs = store.profiles_for(llama3_70b, fake_profile)
    assert len(calls) == 1 and all(p is profs[0] for p in profs)
    store.profiles_for(llama3_8b, fake_profile)
    store.profiles_for(llama31_8b, fake_profile)
    assert calls == [P.attention_key(64, 8, 128), P.attention_key(32, 8, 128)]
    assert len(store) == 2 and store.measured == calls
    assert {k.name() for k in calls} == {"opattn_prefill[64, 8, 128]/bf16", "opattn_prefill[32, 8, 128]/bf16"}
    # a change of head grouping is a different operator
    assert P.attention_key(32, 32, 128) not in store
    assert P.gemm_key(4096, 4096) not in store
    store.get(P.gemm_key(4096, 4096), fake_profile)
    path = str(tmp_path / "profiles.json")
    store.save(path)
    back = P.ProfileStore.load(path)
    assert len(back) == 3 and set(back._profiles) == set(store._profiles)
    q = [[7, 3000], [20, 500]]
    for key in calls:
        np.testing.assert_allclose(back.get(key, None).predict(q), store.get(key, None).predict(q), rtol=0)


def test_llama3_8b_layer_has_five_distinct_operators():
    keys = P.llama3_8b_layer_keys()
    assert len(set(keys.values())) == 5
    store = P.ProfileStore()
    pts = np.array([[1, 128], [1, 8192], [32, 128], [32, 8192]], dtype=float)
    store.profiles_for([k for _ in range(32) for k in keys.values()],
                       lambda key: P.PiecewiseProfile(pts, attention_like(pts)))
    assert len(store.measured) == 5          # 160 operator instances, 5 profiles
