"""Pins of the oracle's budget allocation (Sec. 4.4, Eqs. 9-12, Eq. 5).

Each test checks a property the paper states, or a worked example derived by
hand from the equations (tests/golden/alloc_worked_examples.txt), never the
oracle against itself.
"""
import math
import os
import random

import pytest

from oracle import ripple_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "alloc_worked_examples.txt")


def _golden_cases():
    cases = []
    for line in open(GOLDEN):
        if not line.strip() or line.startswith("#"):
            continue
        name, *kv = line.split()
        d = dict(x.split("=") for x in kv)
        cases.append((name, [float(x) for x in d["s"].split(",")], float(d["r"]),
                      float(d["gamma"]), int(d["B"]), [int(x) for x in d["b"].split(",")]))
    return cases


@pytest.mark.parametrize("case", _golden_cases(), ids=lambda c: c[0])
def test_worked_examples(case):
    _, s, r, gamma, B, expect = case
    assert O.alloc_budgets(s, r, gamma, B) == expect


def _profiles(n=40, seed=7):
    rnd = random.Random(seed)
    out = []
    for _ in range(n):
        L = rnd.choice([1, 2, 3, 4, 7, 32, 80])
        s = [rnd.lognormvariate(-4.0, 1.0) for _ in range(L)]
        r = rnd.choice([1.0, 1.25, 1.5, 1.75, 4.0, 8.0])
        gamma = rnd.choice([math.inf, 0.0, 1.0, 1.5, 2.0, 3.0, 16.0])
        B = rnd.choice([0, 1, L, 10 * L + 3, 128 * L, 1024 * L + 7, 2048 * L])
        out.append((s, r, gamma, B))
    return out


@pytest.mark.parametrize("s,r,gamma,B", _profiles())
def test_budgets_sum_to_global_budget(s, r, gamma, B):
    # Eq. 5: sum_l b_l = B, every b_l a non-negative integer.
    b = O.alloc_budgets(s, r, gamma, B)
    assert sum(b) == B
    assert all(isinstance(x, int) and x >= 0 for x in b)


@pytest.mark.parametrize("L,B", [(1, 5), (3, 10), (4, 512), (32, 32768), (80, 163841)])
def test_identical_sensitivity_is_uniform(L, B):
    # Eq. 9 special case: identical s gives s_hat = 0, hence uniform allocation;
    # leftover tokens go to the lowest layer indices (largest remainder, ties low).
    b = O.alloc_budgets([0.37] * L, 8.0, math.inf, B)
    q, rem = divmod(B, L)
    assert b == [q + 1] * rem + [q] * (L - rem)
    assert O.normalize_sensitivity([0.37] * L) == [0.0] * L


def test_ratio_one_is_uniform():
    # Eq. 10 with r = 1: every multiplier equals one, whatever the profile.
    s = [0.01, 0.5, 0.02, 0.3, 0.7]
    assert O.exponential_map(O.normalize_sensitivity(s), 1.0) == [1.0] * 5
    assert O.alloc_budgets(s, 1.0, math.inf, 500) == [100] * 5


@pytest.mark.parametrize("r", [1.25, 1.5, 4.0, 8.0, 100.0])
def test_max_min_multiplier_ratio_is_r(r):
    # Sec. 4.4: for a nonconstant profile the largest/smallest multiplier ratio
    # before clipping is exactly r (up to the last-place rounding of exp/log).
    s = [0.003, 0.05, 0.011, 0.0524, 0.004]
    wt = O.exponential_map(O.normalize_sensitivity(s), r)
    assert min(wt) == 1.0
    assert max(wt) / min(wt) == pytest.approx(r, rel=2e-15)


def test_normalized_scores_in_unit_interval_and_order_preserving():
    rnd = random.Random(3)
    s = [rnd.random() for _ in range(50)]
    sh = O.normalize_sensitivity(s)
    assert min(sh) == 0.0 and max(sh) == 1.0
    for i in range(50):
        for j in range(50):
            if s[i] < s[j]:
                assert sh[i] <= sh[j]


def test_multipliers_monotone_in_sensitivity():
    # Sec. 4.4: the map is monotone, a more sensitive layer never gets a smaller
    # initial multiplier; budgets then follow up to the one-token rounding.
    rnd = random.Random(11)
    s = [rnd.lognormvariate(-4.0, 1.0) for _ in range(32)]
    wt = O.exponential_map(O.normalize_sensitivity(s), 8.0)
    b = O.alloc_budgets(s, 8.0, math.inf, 32 * 1024)
    order = sorted(range(32), key=lambda i: s[i])
    for a, c in zip(order, order[1:]):
        assert wt[a] <= wt[c]
        assert b[a] <= b[c] + 1


@pytest.mark.parametrize("scale,shift", [(2.0, 0.0), (0.25, 0.0), (1024.0, 0.0)])
def test_exact_affine_invariance(scale, shift):
    # Sec. 4.4: s_hat is invariant to positive affine maps of s. Power-of-two
    # scalings are exact in binary, so the budgets must match exactly.
    s = [0.2, 1.0, 0.6, 0.1, 0.45, 0.33]
    t = [scale * x + shift for x in s]
    assert O.normalize_sensitivity(t) == O.normalize_sensitivity(s)
    assert O.alloc_budgets(t, 4.0, math.inf, 6 * 300) == O.alloc_budgets(s, 4.0, math.inf, 6 * 300)


def test_general_affine_invariance():
    s = [0.2, 1.0, 0.6, 0.1, 0.45, 0.33]
    t = [3.7 * x + 12.5 for x in s]
    for a, c in zip(O.normalize_sensitivity(t), O.normalize_sensitivity(s)):
        assert a == pytest.approx(c, abs=1e-14)


@pytest.mark.parametrize("gamma", [math.inf, 1.0, 1.5, 2.0, 5.0])
def test_clip_normalize_mean_one_and_interval(gamma):
    # Eq. 11: after ClipNormalize the weights have mean one; before the rescale
    # every weight lies in [1/gamma, gamma], so afterwards max/min <= gamma^2.
    s = [0.003, 0.05, 0.011, 0.0524, 0.004, 0.02]
    wt = O.exponential_map(O.normalize_sensitivity(s), 8.0)
    w = O.clip_normalize(wt, gamma)
    assert sum(w) / len(w) == pytest.approx(1.0, abs=4e-15)
    if math.isfinite(gamma):
        assert max(w) / min(w) <= gamma * gamma * (1 + 1e-15)
    else:
        assert max(w) / min(w) == pytest.approx(8.0, rel=4e-15)
    if gamma == 1.0:
        assert w == [1.0] * len(w)


def test_budget_round_half_up_when_consistent():
    # Eq. 12: when independent round-half-up already gives sum B, the
    # reconciled budgets equal it.
    s = [0.2, 1.0, 0.6, 0.1]
    w = O.clip_normalize(O.exponential_map(O.normalize_sensitivity(s), 4.0), math.inf)
    rounded = [math.floor(128 * x + 0.5) for x in w]
    assert sum(rounded) == 512
    assert O.layer_budgets(w, 512) == rounded


def test_keep_count_reading():
    assert O.keep_count(100, 512, 32) == 100
    assert O.keep_count(10, 512, 32) == 32
    assert O.keep_count(5000, 512, 32) == 512
    assert O.keep_count(0, 16, 16) == 16
