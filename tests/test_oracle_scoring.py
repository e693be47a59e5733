"""Pins of the oracle's token scoring, pooling, selection, gather and decoding.

Scoring follows SnapKV's observation-window rule (kept unchanged by RippleKV,
Sec. 4.4 last paragraph); the retained set and compressed cache follow Eq. 4;
decoding follows Sec. 4.1. Pins: closed forms, invariants, library routines
that compute the same special case, and loop-level brute force on tiny inputs.
"""
import math

import numpy as np
import pytest
import scipy.ndimage
import torch

from oracle import ripple_oracle as O


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


# ----------------------------------------------------------------- scoring


def _brute_votes(q_win, k, scale):
    """Loop-level restatement: for every window row, a causal softmax over the
    keys it can see, its probabilities added to the keys' votes."""
    G, w, d = q_win.shape
    T = k.shape[0]
    P = T - w
    votes = [0.0] * T
    for g in range(G):
        for i in range(w):
            seen = range(P + i + 1)
            logit = [sum(q_win[g, i, c] * k[t, c] for c in range(d)) * scale for t in seen]
            m = max(logit)
            z = sum(math.exp(x - m) for x in logit)
            for t in seen:
                votes[t] += math.exp(logit[t] - m) / z
    return np.array(votes)


@pytest.mark.parametrize("G,w,T,d", [(1, 1, 3, 2), (2, 4, 12, 3), (3, 5, 5, 4), (2, 3, 17, 5)])
def test_votes_match_brute_force(G, w, T, d):
    q = _rand((G, w, d), 1 + G + T)
    k = _rand((T, d), 2 + w + d)
    scale = 1.0 / math.sqrt(d)
    votes, _, _ = O.window_votes(q, k, scale)
    np.testing.assert_allclose(votes, _brute_votes(q, k, scale), rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("G,w,T", [(4, 32, 512), (2, 32, 40), (8, 32, 300), (1, 7, 7)])
def test_votes_total_mass(G, w, T):
    # every window row is a probability distribution over keys: total mass G*w
    q = _rand((G, w, 16), 3)
    k = 2.0 * _rand((T, 16), 4)
    votes, _, _ = O.window_votes(q, k, 0.25)
    assert votes.sum() == pytest.approx(G * w, rel=1e-12)
    assert (votes >= 0).all()


@pytest.mark.parametrize("zero_q", [False, True])
def test_votes_identical_keys_closed_form(zero_q):
    # identical keys (or zero queries): each row is uniform over the P+i+1 keys
    # it sees, so prefix key t gets G * sum_i 1/(P+i+1) and window key P+j gets
    # G * sum_{i>=j} 1/(P+i+1).
    G, w, T, d = 4, 32, 512, 64
    P = T - w
    q = np.zeros((G, w, d)) if zero_q else _rand((G, w, d), 5)
    k = np.tile(_rand((1, d), 6), (T, 1))
    votes, _, _ = O.window_votes(q, k, 1.0 / 8.0)
    inv = np.array([1.0 / (P + i + 1) for i in range(w)])
    np.testing.assert_allclose(votes[:P], G * inv.sum(), rtol=1e-12)
    for j in range(w):
        assert votes[P + j] == pytest.approx(G * inv[j:].sum(), rel=1e-12)


def test_causal_mask_isolates_future_window_keys():
    # changing window key P+j must leave rows i < j untouched and move rows i >= j
    G, w, T, d = 2, 8, 40, 8
    P = T - w
    q = _rand((G, w, d), 8)
    k = _rand((T, d), 9)
    j = 5
    k2 = k.copy()
    k2[P + j] = 40.0 * q[0, w - 1] / np.linalg.norm(q[0, w - 1])
    _, m1, s1 = O.window_votes(q, k, 0.3)
    _, m2, s2 = O.window_votes(q, k2, 0.3)
    rows_i = np.tile(np.arange(w), G)
    before = rows_i < j
    np.testing.assert_array_equal(m1[before], m2[before])
    np.testing.assert_array_equal(s1[before], s2[before])
    assert not np.allclose(s1[~before] * np.exp(m1[~before]), s2[~before] * np.exp(m2[~before]))


def test_scale_enters_logits():
    # with scale s the votes equal unscaled votes of queries multiplied by s
    q = _rand((2, 4, 6), 10)
    k = _rand((20, 6), 11)
    a, _, _ = O.window_votes(q, k, 0.37)
    b, _, _ = O.window_votes(0.37 * q, k, 1.0)
    np.testing.assert_allclose(a, b, rtol=1e-12)


def test_gqa_group_rows_are_summed():
    # the votes of a group are the sum of the single-head votes of its members
    q = _rand((3, 5, 4), 12)
    k = _rand((30, 4), 13)
    total, _, _ = O.window_votes(q, k, 0.5)
    parts = sum(O.window_votes(q[g:g + 1], k, 0.5)[0] for g in range(3))
    np.testing.assert_allclose(total, parts, rtol=1e-12)


# ----------------------------------------------------------------- pooling


@pytest.mark.parametrize("P,kernel", [(1, 7), (5, 7), (6, 7), (100, 7), (100, 3), (33, 1)])
def test_max_pool_matches_scipy(P, kernel):
    # edge-replicating padding never changes a max, so scipy's
    # maximum_filter1d(mode="nearest") equals the clipped-window max
    x = np.random.default_rng(P).random(P).astype(np.float32)
    ref = scipy.ndimage.maximum_filter1d(x, size=kernel, mode="nearest")
    np.testing.assert_array_equal(O.pool_scores(x, kernel, "max"), ref)


def test_max_pool_one_hot_is_box():
    x = np.zeros(50, np.float32)
    x[20] = 1.0
    x[1] = 0.5
    out = O.pool_scores(x, 7, "max")
    expect = np.zeros(50, np.float32)
    expect[0:5] = 0.5
    expect[17:24] = 1.0
    np.testing.assert_array_equal(out, expect)


def test_avg_pool_clipped_window_mean():
    x = np.random.default_rng(1).random(64).astype(np.float32)
    out = O.pool_scores(x, 7, "avg")
    c = np.concatenate([[0.0], np.cumsum(x.astype(np.float64))])
    lo = np.maximum(np.arange(64) - 3, 0)
    hi = np.minimum(np.arange(64) + 4, 64)
    ref = (c[hi] - c[lo]) / (hi - lo)
    np.testing.assert_allclose(out, ref, rtol=2e-6)
    const = np.full(20, 0.25, np.float32)
    np.testing.assert_array_equal(O.pool_scores(const, 7, "avg"), const)


# ----------------------------------------------------------------- selection


def _check_topk(pooled, idx, n, T, w):
    P = T - w
    K = n - w
    assert len(idx) == n
    assert list(idx) == sorted(set(idx.tolist()))
    assert list(idx[K:]) == list(range(P, T))
    kept = set(idx[:K].tolist())
    assert all(0 <= t < P for t in kept)
    dropped = [t for t in range(P) if t not in kept]
    for a in kept:
        for b in dropped:
            assert pooled[a] > pooled[b] or (pooled[a] == pooled[b] and a < b)


@pytest.mark.parametrize("seed", range(6))
def test_selection_is_top_k_with_low_index_ties(seed):
    rnd = np.random.default_rng(seed)
    T, w = int(rnd.integers(40, 120)), int(rnd.integers(1, 9))
    P = T - w
    pooled = (rnd.integers(0, 12, P) / 8.0).astype(np.float32)  # many ties
    n = int(rnd.integers(w, T + 1))
    idx = O.select_tokens(pooled, n, T, w)
    _check_topk(pooled, idx, n, T, w)


def test_selection_all_equal_keeps_lowest_indices():
    T, w, n = 100, 8, 30
    idx = O.select_tokens(np.ones(92, np.float32), n, T, w)
    assert list(idx) == list(range(22)) + list(range(92, 100))


def test_selection_keep_all_and_window_only():
    pooled = np.random.default_rng(0).random(50).astype(np.float32)
    assert list(O.select_tokens(pooled, 58, 58, 8)) == list(range(58))
    assert list(O.select_tokens(pooled, 8, 58, 8)) == list(range(50, 58))


# ----------------------------------------------------------------- compress


def test_compress_unit_keep_all_is_identity():
    q = _rand((2, 4, 8), 1)
    k = _rand((64, 8), 2)
    v = _rand((64, 8), 3)
    out = O.compress_unit(q, k, v, budget=1000, w=4, scale=0.35)
    assert list(out["idx"]) == list(range(64))
    np.testing.assert_array_equal(out["k_out"], k)
    np.testing.assert_array_equal(out["v_out"], v)


def test_compress_unit_gathers_selected_rows():
    q = _rand((2, 4, 8), 4)
    k = _rand((64, 8), 5)
    v = _rand((64, 8), 6)
    out = O.compress_unit(q, k, v, budget=20, w=4, scale=0.35)
    _check_topk(out["pooled"], out["idx"], 20, 64, 4)
    np.testing.assert_array_equal(out["k_out"], k[out["idx"]])
    np.testing.assert_array_equal(out["v_out"], v[out["idx"]])


# ----------------------------------------------------------------- decoding


@pytest.mark.parametrize("G,n,d", [(4, 1, 64), (4, 37, 64), (8, 300, 128), (2, 2, 16)])
def test_decode_matches_torch_sdpa(G, n, d):
    q = _rand((G, d), n)
    k = _rand((n, d), n + 1)
    v = _rand((n, d), n + 2)
    scale = 1.0 / math.sqrt(d)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q)[:, None, :], torch.from_numpy(k)[None].expand(G, n, d),
        torch.from_numpy(v)[None].expand(G, n, d), scale=scale)[:, 0, :].numpy()
    np.testing.assert_allclose(O.decode_attention(q, k, v, scale), ref, rtol=1e-12, atol=1e-13)


def test_decode_closed_forms():
    q = _rand((4, 32), 1)
    v = _rand((1, 32), 2)
    np.testing.assert_allclose(O.decode_attention(q, _rand((1, 32), 3), v, 0.2), np.tile(v, (4, 1)))
    k = np.tile(_rand((1, 32), 4), (9, 1))
    v9 = _rand((9, 32), 5)
    np.testing.assert_allclose(O.decode_attention(q, k, v9, 0.2), np.tile(v9.mean(0), (4, 1)),
                               rtol=1e-12, atol=1e-14)


# ------------------------------------------- window rows' prefill attention


@pytest.mark.parametrize("G,w,T,d", [(1, 1, 1, 4), (2, 4, 12, 3), (4, 32, 300, 16), (8, 7, 7, 5)])
def test_window_attention_matches_torch_sdpa(G, w, T, d):
    # the window rows of a causal prefill attention: torch's scaled dot-product
    # attention over all T queries with its own causal mask, last w rows taken
    rng = np.random.default_rng(7 + G + T)
    q_all = rng.standard_normal((G, T, d))
    k = 2.0 * rng.standard_normal((T, d))
    v = rng.standard_normal((T, d))
    scale = 1.0 / math.sqrt(d)
    got = O.window_attention(q_all[:, T - w:], k, v, scale)
    t = lambda a: torch.from_numpy(a)
    ref = torch.nn.functional.scaled_dot_product_attention(
        t(q_all)[None], t(k)[None, None].expand(1, G, T, d), t(v)[None, None].expand(1, G, T, d),
        is_causal=True, scale=scale)[0, :, T - w:].numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-13)


def test_window_attention_closed_forms():
    G, w, T, d = 2, 5, 9, 4
    P = T - w
    rng = np.random.default_rng(11)
    q = rng.standard_normal((G, w, d))
    v = rng.standard_normal((T, d))
    # identical keys: row i averages the P + i + 1 values it can see
    k = np.tile(rng.standard_normal(d), (T, 1))
    got = O.window_attention(q, k, v, 0.5)
    for i in range(w):
        np.testing.assert_allclose(got[:, i], np.tile(v[:P + i + 1].mean(0), (G, 1)), rtol=1e-12)
    # one token: the value itself
    one = O.window_attention(q[:, :1], k[:1], v[:1], 0.5)
    np.testing.assert_allclose(one, np.tile(v[0], (G, 1, 1)), rtol=0, atol=0)
    # the row's probabilities are those the votes add up: with one-hot value
    # columns the output is the row's attention over the keys, and its sum
    # over rows is the vote of every key
    kk = rng.standard_normal((T, d))
    votes, _, _ = O.window_votes(q, kk, 0.5)
    probs = O.window_attention(q, kk, np.eye(T), 0.5)
    assert probs.shape == (G, w, T)
    np.testing.assert_allclose(probs.sum(axis=2), 1.0, rtol=1e-12)
    np.testing.assert_allclose(probs.sum(axis=(0, 1)), votes, rtol=1e-12)
    # the causal mask: a row never weights a later window token
    for i in range(w):
        assert np.all(probs[:, i, P + i + 1:] == 0)
