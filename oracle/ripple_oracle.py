"""CPU oracle for the RippleKV serving path (arxiv 2608.08684).

TEST INFRASTRUCTURE ONLY. Only the test suite, the smoke check and the
benchmark's CPU-baseline leg may import this module. The product (the CUDA
library and its Python binding) never calls it, and this module imports
nothing from the product.

Plain, slow and meant to be read against the paper: every function follows one
passage, in the paper's order and notation, in float64 (Python floats / numpy
float64) unless noted. Library primitives used as single steps: numpy matmul,
exp, max, sum and a stable lexicographic sort.

Paper passages followed:
  * Sec. 4.1 (problem formulation): the per-layer cache C_l, the retained set
    S_l, the compressed cache (Eq. 4) and the global budget sum_l b_l = B (Eq. 5).
  * Sec. 4.4 / Algorithm 1 "Budget Allocation": Eq. 9 (min-max normalisation,
    identical sensitivities give s_hat = 0), Eq. 10 (exponential map r^s_hat),
    Eq. 11 (ClipNormalize to [1/gamma, gamma], then mean one), Eq. 12
    (b_l = round(B/|A| w_l)).
  * Sec. 4.4, last paragraph: RippleKV keeps the SnapKV token scoring and
    selection rule and only changes b_l. SnapKV (Sec. 2) scores prompt tokens
    from an observation window at the end of the prompt.
  * Sec. 4.1: during decoding each new query attends to the cached states.
  * Sec. 4.3 (sensitivity profiling, offline): the norm-adaptive Value
    perturbation (Eq. 6), the output KL averaged over the evaluation window
    (Eq. 7) and the average over the calibration set (Eq. 8).

Readings where the paper is silent (each is also listed in the design notes):
  R1 Eq. 9 without the +epsilon of Algorithm 1: the only role of epsilon is
     the identical-sensitivity case, which Eq. 9 handles explicitly, and the
     stated "max/min multiplier is exactly r" only holds without it.
  R2 gamma <= 0 or infinite means "no clipping" (the paper gives no value);
     one clip, then one rescale to mean one (Eq. 11), no iteration.
  R3 round() in Eq. 12 cannot keep Eq. 5 exact in general; we use floor plus
     largest remainder (ties to the lower layer index), which equals
     round-half-up whenever that already sums to B.
  R4 b_l counts the observation window; each (batch, kv head) of layer l keeps
     n_l = min(T, max(b_l, w)) tokens: the w window tokens plus the top
     n_l - w prefix tokens.
  R5 scoring: window query rows r = (query head g of the KV head's GQA group,
     window position i), query position P + i with P = T - w; logits
     q.k * scale (scale = 1/sqrt(d)), causal inside the window (row i sees
     keys t <= P + i), softmax over all visible keys, vote of key t =
     sum over all rows of the softmax probability.
  R6 pooling over the prefix votes, kernel k (odd), stride 1, window clipped
     to the prefix: max-pool (default) or average over the clipped window.
  R7 selection by (pooled score descending, token index ascending); retained
     indices emitted in ascending order, window last.
  R8 decisions on scores are taken in fp32, the precision the kernels score
     in: the fp64 votes are rounded to fp32 before pooling and selection.
  R9 decoding: the new key/value row is appended first and the new query
     attends to it as well (causal self-inclusion); no positional rotation
     (the synthetic keys stand for post-rotation keys).
  R10 perturbation (Eq. 6): the positions the base method protects (SnapKV's
     observation window) are left out by the caller through a position
     range [pos_begin, pos_end) of eligible rows; the draws eps ~ N(0, I) are
     an input (one d-vector per eligible row), not drawn here.
  R11 window KL (Eq. 7): P_t and Q_t are the softmax over the vocabulary of
     the reference and perturbed logits at window position t; logits are
     finite.

Parity pins (tests/test_oracle_*.py): allocation invariants the paper states
(sum = B, uniform profile, r = 1, max/min = r, monotonicity, affine
invariance, mean-one weights, clip interval) and a hand-derived worked
example; scoring closed forms (identical keys, probability mass per row),
causal-mask isolation and a loop-level brute force on tiny inputs; pooling
against scipy's maximum_filter1d; selection against the defining top-k
property; decoding against torch's scaled_dot_product_attention and the
len-1 / identical-key closed forms; perturbation against the one-hot closed
form and the noise-norm identity; window KL against the two-category and
uniform-versus-spike closed forms, KL(P||P) = 0 and shift invariance. The end-to-end quality of the method on
LongBench is parity unpinned (no model weights or dataset here).
"""
from __future__ import annotations

import math

import numpy as np

# ---------------------------------------------------------------------------
# Budget allocation: Sec. 4.4, Eqs. 9-12, Algorithm 1 "Budget Allocation".
# Plain Python floats (IEEE double) and libm exp/log, layer order throughout.
# ---------------------------------------------------------------------------


def normalize_sensitivity(s):
    """Eq. 9: s_hat_l = (s_l - s_min) / (s_max - s_min); all identical -> 0 (reading R1)."""
    s_min = s[0]
    s_max = s[0]
    for x in s:
        if x < s_min:
            s_min = x
        if x > s_max:
            s_max = x
    if s_max == s_min:
        return [0.0 for _ in s]
    span = s_max - s_min
    return [(x - s_min) / span for x in s]


def exponential_map(s_hat, r):
    """Eq. 10: w_tilde_l = exp(log r * s_hat_l) = r ** s_hat_l, r >= 1."""
    log_r = math.log(r)
    return [math.exp(log_r * x) for x in s_hat]


def clip_normalize(w_tilde, gamma):
    """Eq. 11: clip to [1/gamma, gamma] (gamma >= 1), then rescale to mean one (reading R2)."""
    clip = gamma > 0.0 and math.isfinite(gamma)
    if clip:
        lo = 1.0 / gamma
        c = [min(max(x, lo), gamma) for x in w_tilde]
    else:
        c = list(w_tilde)
    total = 0.0
    for x in c:
        total += x
    mean = total / len(c)
    return [x / mean for x in c]


def layer_budgets(w, B):
    """Eq. 12, b_l = round(B/|A| * w_l), reconciled so that Eq. 5 holds exactly (reading R3).

    floor of every quota, then one extra token to each of the B - sum(floor)
    layers with the largest fractional parts, ties to the lower layer index.
    """
    n = len(w)
    avg = B / n
    quota = [avg * x for x in w]
    base = [math.floor(x) for x in quota]
    frac = [quota[i] - base[i] for i in range(n)]
    left = B - sum(base)
    order = sorted(range(n), key=lambda i: (-frac[i], i))
    for i in order[:left]:
        base[i] += 1
    return [int(x) for x in base]


def alloc_budgets(s, r, gamma, B):
    """Algorithm 1 "Budget Allocation": s -> s_hat -> w_tilde -> w -> b."""
    return layer_budgets(clip_normalize(exponential_map(normalize_sensitivity(s), r), gamma), B)


def keep_count(b, T, w):
    """Tokens kept per (batch, kv head) of a layer with budget b (reading R4)."""
    return min(T, max(int(b), w))


# ---------------------------------------------------------------------------
# Token scoring and selection: SnapKV's observation-window rule, kept
# unchanged by RippleKV (Sec. 4.4 last paragraph; Sec. 2).
# One "unit" = one (batch, layer, kv head).
# ---------------------------------------------------------------------------


def window_votes(q_win, k, scale):
    """Vote of every key of one unit (readings R5).

    q_win: [G][w][d] window queries of the G query heads that share this KV head.
    k:     [T][d] keys of this KV head.
    Returns (votes [T], row_max [G*w], row_sum [G*w]) in float64: votes[t] is
    the softmax probability mass key t receives, summed over all window rows.
    """
    G, w, d = q_win.shape
    T = k.shape[0]
    P = T - w
    rows = q_win.reshape(G * w, d)
    logits = (rows @ k.T) * scale
    row_pos = P + np.tile(np.arange(w), G)
    visible = np.arange(T)[None, :] <= row_pos[:, None]
    logits = np.where(visible, logits, -np.inf)
    row_max = logits.max(axis=1)
    e = np.exp(logits - row_max[:, None])
    row_sum = e.sum(axis=1)
    probs = e / row_sum[:, None]
    return probs.sum(axis=0), row_max, row_sum


def window_attention(q_win, k, v, scale):
    """Prefill attention output of the observation-window rows of one unit
    (the rows whose softmax SnapKV's scoring reads, reading R5; computed here
    directly from that definition, with the same causal mask).

    q_win: [G][w][d]; k, v: [T][d]. Returns [G][w][d] float64: row (g, i), at
    token P + i, is sum over keys t <= P + i of softmax_t(scale q . k_t) v_t.
    """
    G, w, d = q_win.shape
    T = k.shape[0]
    P = T - w
    out = np.zeros((G, w, v.shape[1]))
    for g in range(G):
        for i in range(w):
            vis = P + i + 1
            logits = (k[:vis] @ q_win[g, i]) * scale
            e = np.exp(logits - logits.max())
            out[g, i] = (e / e.sum()) @ v[:vis]
    return out


def pool_scores(votes, kernel, kind="max"):
    """1-D pooling of the prefix votes (reading R6), in the dtype of `votes`.

    max: out[t] = max of votes[j] over |j - t| <= kernel//2, 0 <= j < P.
    avg: the same window summed in ascending j from zero, divided by its size.
    none: votes unchanged.
    """
    P = votes.shape[0]
    half = kernel // 2
    if kind == "none" or kernel <= 1 or P == 0:
        return votes.copy()
    out = np.empty_like(votes)
    for t in range(P):
        lo = max(0, t - half)
        hi = min(P, t + half + 1)
        if kind == "max":
            out[t] = votes[lo:hi].max()
        elif kind == "avg":
            acc = votes.dtype.type(0)
            for j in range(lo, hi):
                acc = votes.dtype.type(acc + votes[j])
            out[t] = votes.dtype.type(acc / votes.dtype.type(hi - lo))
        else:
            raise ValueError(kind)
    return out


def select_tokens(pooled, n_keep, T, w):
    """Retained positions S_l of one unit (Eq. 4; reading R7).

    The n_keep - w prefix tokens with the largest pooled score (ties: lower
    index first) plus the w window tokens, in ascending order.
    """
    P = T - w
    n_prefix = n_keep - w
    order = np.lexsort((np.arange(P), -pooled))
    kept = np.sort(order[:n_prefix])
    return np.concatenate([kept, np.arange(P, T)]).astype(np.int64)


def compress_unit(q_win, k, v, budget, w, scale, pool_kernel=7, pool_kind="max"):
    """Compress one (batch, layer, kv head): score, pool, select, gather (Eq. 4).

    Returns dict(idx, k_out, v_out, votes (prefix, float64), pooled (fp32)).
    """
    T = k.shape[0]
    n = keep_count(budget, T, w)
    P = T - w
    out = {}
    if n >= T:
        idx = np.arange(T, dtype=np.int64)
        out["votes"] = window_votes(q_win, k, scale)[0][:P] if P > 0 else np.zeros(0)
        out["pooled"] = None
    else:
        votes = window_votes(q_win, k, scale)[0][:P]
        pooled = pool_scores(votes.astype(np.float32), pool_kernel, pool_kind)
        idx = select_tokens(pooled, n, T, w)
        out["votes"] = votes
        out["pooled"] = pooled
    out["idx"] = idx
    out["k_out"] = k[idx]
    out["v_out"] = v[idx]
    return out


# ---------------------------------------------------------------------------
# Decoding against the compressed cache (Sec. 4.1; reading R9).
# ---------------------------------------------------------------------------


def decode_attention(q, k_rows, v_rows, scale):
    """o_g = softmax(q_g . k_j * scale over rows j) weighted sum of v_j.

    q: [G][d]; k_rows, v_rows: [n][d], the retained rows followed by the
    appended rows, the current token's row last. Returns [G][d] float64.
    """
    logits = (q @ k_rows.T) * scale
    m = logits.max(axis=1, keepdims=True)
    e = np.exp(logits - m)
    return (e @ v_rows) / e.sum(axis=1, keepdims=True)


# ---------------------------------------------------------------------------
# Sensitivity profiling, offline (Sec. 4.3, Eqs. 6-8; readings R10, R11).
# The model forwards between the perturbation and the KL (the "PerturbedPredict"
# and "ReferencePredict" steps of Algorithm 1) are not part of this oracle.
# ---------------------------------------------------------------------------


def perturb_values(v, eps, alpha, pos_begin, pos_end):
    """Eq. 6: v~_u = v_u + alpha * ||v_u||_2 * eps_u for every (batch, kv head)
    and every eligible position u in [pos_begin, pos_end); all other rows are
    returned unchanged (reading R10).

    v: [B][Hkv][T][d] the layer's Value cache; eps: [B][Hkv][pos_end - pos_begin][d]
    the standard normal draws, eps[b, h, u - pos_begin] for position u.
    Returns a float64 copy of v with the eligible rows perturbed.
    """
    out = np.array(v, dtype=np.float64, copy=True)
    rows = out[:, :, pos_begin:pos_end, :]
    norm = np.sqrt(np.sum(rows * rows, axis=-1, keepdims=True))  # ||v_u||_2 per row
    out[:, :, pos_begin:pos_end, :] = rows + alpha * norm * np.asarray(eps, dtype=np.float64)
    return out


def log_softmax(x):
    """log of the softmax over the last axis: x - (m + log sum exp(x - m))."""
    x = np.asarray(x, dtype=np.float64)
    m = x.max(axis=-1, keepdims=True)
    return x - (m + np.log(np.sum(np.exp(x - m), axis=-1, keepdims=True)))


def window_kl(p_logits, q_logits):
    """Eq. 7: d = (1/|W|) sum over window positions t of KL(P_t || Q_t), with
    P_t = softmax(p_logits[t]) the reference distribution and Q_t =
    softmax(q_logits[t]) the distribution after the perturbation (reading R11).

    p_logits, q_logits: [|W|][V]. Returns (kl [|W|], d), float64.
    """
    log_p = log_softmax(p_logits)
    log_q = log_softmax(q_logits)
    kl = np.sum(np.exp(log_p) * (log_p - log_q), axis=-1)
    return kl, float(np.mean(kl))


def sensitivity_profile(d):
    """Eq. 8: s_l = (1/N) sum_i d_{i,l}; d: [N][|A|] window responses of the N
    calibration examples for every compressible layer. Returns [|A|] float64,
    summed in example order."""
    d = np.asarray(d, dtype=np.float64)
    s = np.zeros(d.shape[1])
    for i in range(d.shape[0]):
        s = s + d[i]
    return s / d.shape[0]
