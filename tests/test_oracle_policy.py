"""Pins for the oracle's allocation policy (Sec. 4.2, Eq. 6-8; Sec. 4.3, Eq. 9).

The normalizer reading (multiplicative rescale, then clip to [0,1], mean
equal to the target) is pinned two ways: against an exact piecewise-linear
inversion written here, and against the "High" step counts of Table D, which
the policy can only produce if every per-step budget lies inside the
envelope that this reading gives.  An additive-shift reading of the
normalizer is shown to contradict Table D.
"""
import os

import numpy as np
import pytest

import oracle

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def read_table(name):
    rows = []
    for line in open(os.path.join(GOLD, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            rows.append(line.split())
    return rows


def settings():
    return {r[0]: dict(T=int(r[1]), orient=r[2], B=float(r[3]), rho=float(r[4]), alpha=float(r[5]))
            for r in read_table("sec5_policy_defaults.txt")}


def demand_prior():
    return {r[0]: float(r[1]) for r in read_table("table_a_demand_prior.txt")}


def test_profile_closed_form_and_symmetry():
    for T in (1, 16, 32, 7):
        early = oracle.policy_profile(T, "early")
        late = oracle.policy_profile(T, "late")
        t = np.arange(1, T + 1)
        np.testing.assert_allclose(early, 1 - (t - 0.5) / T, rtol=0, atol=1e-15)
        np.testing.assert_allclose(late, early[::-1], rtol=0, atol=1e-15)
        assert (early > 0).all() and (early < 1).all()  # no zero endpoints
        np.testing.assert_allclose(early.mean(), 0.5, atol=1e-15)


def exact_normalize(p, target):
    """Exact inversion of mean(clip(s p, 0, 1)) = target over the number m of
    steps clipped at 1 (the m largest entries of p)."""
    p = np.asarray(p, float)
    T = p.size
    order = np.argsort(-p, kind="stable")
    ps = p[order]
    for m in range(T + 1):
        rest = ps[m:].sum()
        if rest <= 0:
            s = np.inf
        else:
            s = (T * target - m) / rest
        if s < 0:
            continue
        ok_top = m == 0 or s * ps[m - 1] >= 1 - 1e-12
        ok_rest = m == T or s * ps[m] <= 1 + 1e-12
        if ok_top and ok_rest:
            return np.clip(s * p, 0, 1)
    raise AssertionError("no consistent clip set")


@pytest.mark.parametrize("T,orient", [(16, "early"), (32, "late"), (9, "early")])
@pytest.mark.parametrize("target", [0.1, 0.36, 0.45, 0.6, 0.75, 0.9])
def test_normalizer_matches_exact_inversion(T, orient, target):
    p = oracle.policy_profile(T, orient)
    got = oracle.policy_normalize(p, target)
    np.testing.assert_allclose(got, exact_normalize(p, target), rtol=0, atol=1e-12)
    np.testing.assert_allclose(got.mean(), target, atol=1e-12)
    assert (got >= 0).all() and (got <= 1).all()
    # phase ordering is preserved
    order = np.argsort(p)
    assert (np.diff(got[order]) >= -1e-15).all()


def test_normalizer_edge_targets():
    p = oracle.policy_profile(8, "late")
    np.testing.assert_array_equal(oracle.policy_normalize(p, 0.0), np.zeros(8))
    np.testing.assert_array_equal(oracle.policy_normalize(p, 1.0), np.ones(8))
    np.testing.assert_array_equal(oracle.policy_normalize(p, 1.5), np.ones(8))


def test_llada_v_lower_trajectory_closed_form():
    # T=16, early, lower target (1-rho)B = 0.6: the three largest entries
    # clip at 1, the rest are s p_t with s = (16*0.6 - 3) / sum(p_4..p_16)
    s = settings()["llada_v"]
    p = oracle.policy_profile(s["T"], s["orient"])
    lo, _ = oracle.policy_envelope(p, s["B"], s["rho"], 1.0)
    scale = (16 * 0.6 - 3) / p[3:].sum()
    np.testing.assert_allclose(lo, np.concatenate([[1, 1, 1], scale * p[3:]]), atol=1e-12)
    views = [oracle.policy_view(b) for b in lo]
    assert views == [2] * 7 + [1] * 5 + [0] * 4


def test_risk_and_interpolation_special_cases():
    assert oracle.policy_risk(1, 1.0, 0.9, 0.0) == 1.0  # r_1 = 1
    assert oracle.policy_risk(5, 0.0, 0.9, 0.1) == 1.0  # alpha = 0
    assert oracle.policy_risk(5, 1.0, 1.0, 0.0) == 0.0  # confident and stable
    assert oracle.policy_risk(5, 1.0, 1.0, 1.0) == 1.0  # full churn
    assert abs(oracle.policy_risk(3, 0.5, 0.8, 0.25) - (1 - 0.5 * 0.8 * 0.75)) < 1e-15
    assert oracle.policy_budget(0.2, 0.7, 0.0) == 0.2
    assert oracle.policy_budget(0.2, 0.7, 1.0) == 0.7
    assert abs(oracle.policy_budget(0.2, 0.7, 0.5) - 0.45) < 1e-15


def test_thirds_quantization():
    assert oracle.policy_view(0.0) == 0
    assert oracle.policy_view(np.nextafter(1 / 3, 0)) == 0
    assert oracle.policy_view(1 / 3) == 1
    assert oracle.policy_view(np.nextafter(2 / 3, 0)) == 1
    assert oracle.policy_view(2 / 3) == 2
    assert oracle.policy_view(1.0) == 2


def test_budget_stays_in_envelope_and_mean_below_B():
    rng = np.random.default_rng(0)
    for name, s in settings().items():
        p = oracle.policy_profile(s["T"], s["orient"])
        for d in demand_prior().values():
            lo, up = oracle.policy_envelope(p, s["B"], s["rho"], d)
            assert (lo <= up + 1e-15).all()
            assert up.mean() <= s["B"] + 1e-12
            for _ in range(20):
                cbar = rng.random(s["T"])
                chi = rng.random(s["T"])
                b = []
                for t in range(1, s["T"] + 1):
                    r = oracle.policy_risk(t, s["alpha"], cbar[t - 2] if t > 1 else 0.0,
                                           chi[t - 2] if t > 2 else 0.0)
                    assert 0 <= r <= 1
                    b.append(oracle.policy_budget(lo[t - 1], up[t - 1], r))
                b = np.array(b)
                assert (b >= lo - 1e-15).all() and (b <= up + 1e-15).all()
                assert b.mean() <= s["B"] + 1e-12


def high_count(b):
    return sum(oracle.policy_view(x) == 2 for x in b)


def test_table_d_high_step_counts_lie_in_the_reachable_range():
    st = settings()
    prior = demand_prior()
    for backbone, _bench, demand, value in read_table("table_d_high_steps.txt"):
        s = st[backbone]
        value = float(value)
        p = oracle.policy_profile(s["T"], s["orient"])
        ds = [1.0] if demand == "uniform" else list(prior.values())
        lo_counts, hi_counts = [], []
        for d in ds:
            lo, up = oracle.policy_envelope(p, s["B"], s["rho"], d)
            # r_t ranges over [1 - alpha, 1] (cbar, chi in [0,1]); r_1 = 1
            r_min = 1 - s["alpha"]
            lo_counts.append(high_count(lo + r_min * (up - lo)))
            hi_counts.append(high_count(up))
        assert min(lo_counts) <= value <= max(hi_counts), (backbone, demand, value, lo_counts, hi_counts)


def test_additive_shift_reading_contradicts_table_d():
    # N(p; target) read as clip(p + c, 0, 1): LaViDa's lower trajectory alone
    # already has more High steps than the default's average in Table D, and
    # budgets never fall below the lower trajectory.
    s = settings()["lavida"]
    p = oracle.policy_profile(s["T"], s["orient"])
    target = (1 - s["rho"]) * s["B"]
    lo_c, hi_c = -1.0, 1.0
    for _ in range(200):
        c = 0.5 * (lo_c + hi_c)
        if np.clip(p + c, 0, 1).mean() < target:
            lo_c = c
        else:
            hi_c = c
    lower_shift = np.clip(p + 0.5 * (lo_c + hi_c), 0, 1)
    defaults = [float(v) for bb, _b, d, v in read_table("table_d_high_steps.txt")
                if bb == "lavida" and d == "default"]
    assert high_count(lower_shift) > max(defaults)
    # the multiplicative reading stays consistent
    lo, _ = oracle.policy_envelope(p, s["B"], s["rho"], 1.0)
    assert high_count(lo) <= min(defaults)
