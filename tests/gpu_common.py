"""Helpers of the GPU parity tests: run the C-ABI path on seeded inputs and
compare it with the CPU oracle on the same inputs."""
from __future__ import annotations

import numpy as np
import torch

from oracle import ripple_oracle as O
from paper_2608_08684_gb300 import synth

SCORE_RTOL = 1e-3      # votes: relative, fp32 accumulation from bf16/fp32 inputs
SCORE_ATOL_REL = 1e-9  # absolute floor, relative to the largest vote (underflow guard)
SELECT_GAP_RTOL = 2e-3  # a set mismatch needs two votes within 2x the score tolerance
DECODE_ATOL = 2e-2     # decode output, max-abs against the fp64 oracle (acceptance bar)
# Decode output, max-abs: the kernel's own precision, for values of unit scale
# (every test draws or normalises them so). Inputs are exact in fp32;
# each lane sums its share of a group's rows (at most a few hundred terms of
# |p v| <= |v|, |v| < 6) in fp32 and the shares merge through short trees, with
# exponentials of relative error ~2^-22: a worst case of a few 1e-5, observed
# ~1e-6. Dropping or repeating one row of an n-row cache moves the output by
# about 1/n (a few 1e-4 at the lengths tested), so this bound sees it where
# the acceptance bar does not.
DECODE_PREC_ATOL = 1e-4


def layer_inputs(wl, layer, device):
    """(q_win, k, v) of one layer, generated on `device`."""
    return (synth.layer_window_queries(wl, layer, device), synth.layer_keys(wl, layer, device),
            synth.layer_values(wl, layer, device))


def run_compress(lib, wl, budget, q_win, k, v, cap_extra=0, scores=True, pool="max", scale=0.0):
    """ripple_compress_layer on device tensors; returns a dict of device outputs."""
    dev = k.device
    desc = lib.layer_desc(wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.seq_len,
                          wl.window, wl.pool_kernel, pool, wl.torch_dtype, scale)
    n = lib.ripple_keep_count(budget, wl.seq_len, wl.window)
    cap = n + cap_extra
    B, H, d, P = wl.batch, wl.n_kv_heads, wl.head_dim, wl.seq_len - wl.window
    out = {
        "k_out": torch.zeros(B, H, cap, d, dtype=wl.torch_dtype, device=dev),
        "v_out": torch.zeros(B, H, cap, d, dtype=wl.torch_dtype, device=dev),
        "idx": torch.full((B * H * n,), -1, dtype=torch.int32, device=dev),
        "scores": torch.zeros(B, H, P, dtype=torch.float32, device=dev) if scores else None,
        "ws": torch.empty(lib.ripple_compress_workspace_bytes(desc), dtype=torch.uint8,
                          device=dev),
        "status": torch.zeros(1, dtype=torch.int32, device=dev),
    }
    got = lib.ripple_compress_layer(desc, budget, q_win, k, v, out["k_out"], out["v_out"],
                                    out["idx"], out["ws"], scores_out=out["scores"],
                                    dev_status=out["status"])
    torch.cuda.synchronize()
    assert got == n
    out["n"] = n
    out["idx"] = out["idx"].view(B, H, n)
    return out


def unit_f64(wl, q_win, k, v, b, h):
    """float64 copies of one unit's window queries [G][w][d], keys and values [T][d]."""
    G = wl.group
    return (synth.to_f64(q_win[b, h * G:(h + 1) * G]), synth.to_f64(k[b, h]), synth.to_f64(v[b, h]))


def assert_votes_close(gpu, ref):
    gpu = np.asarray(gpu, np.float64)
    err = np.abs(gpu - ref)
    bound = SCORE_RTOL * np.abs(ref) + SCORE_ATOL_REL * (ref.max() if ref.size else 0.0)
    bad = np.nonzero(err > bound)[0]
    assert bad.size == 0, f"{bad.size} votes out of tolerance, first {bad[:5]} " \
                          f"gpu {gpu[bad[:5]]} oracle {ref[bad[:5]]}"


def selection_mismatch(gpu_idx, ora_idx, ora_pooled, n, w):
    """(agreeing prefix tokens, prefix tokens) after checking that every set
    difference lies within the score tolerance of the oracle's threshold."""
    K = n - w
    if K <= 0:
        return 0, 0
    g = set(np.asarray(gpu_idx[:K]).tolist())
    o = set(np.asarray(ora_idx[:K]).tolist())
    tau = float(np.sort(ora_pooled.astype(np.float64))[::-1][K - 1])
    for t in g ^ o:
        assert abs(float(ora_pooled[t]) - tau) <= SELECT_GAP_RTOL * tau, \
            f"token {t} differs with pooled {ora_pooled[t]} vs threshold {tau}"
    return len(g & o), K


def check_compress_unit(wl, out, q_win, k, v, b, h, budget, pool="max", scale=None):
    """Oracle comparison of one unit; returns (agreeing, total) prefix selections."""
    q, kk, vv = unit_f64(wl, q_win, k, v, b, h)
    scale = scale or 1.0 / np.sqrt(wl.head_dim)
    ref = O.compress_unit(q, kk, vv, budget, wl.window, scale, wl.pool_kernel, pool)
    n = out["n"]
    gidx = out["idx"][b, h].cpu().numpy()
    # structure of the retained set (Eq. 4)
    assert len(gidx) == n
    assert np.all(np.diff(gidx) > 0) and gidx[0] >= 0 and gidx[-1] < wl.seq_len
    assert list(gidx[n - wl.window:]) == list(range(wl.seq_len - wl.window, wl.seq_len))
    # gather: retained rows byte-identical to the inputs at the kept positions
    sel = torch.from_numpy(gidx.astype(np.int64)).to(k.device)
    assert torch.equal(out["k_out"][b, h, :n], k[b, h].index_select(0, sel))
    assert torch.equal(out["v_out"][b, h, :n], v[b, h].index_select(0, sel))
    if out["scores"] is not None and wl.seq_len > wl.window:
        assert_votes_close(out["scores"][b, h].cpu().numpy(), ref["votes"])
    if n == wl.seq_len:
        assert list(gidx) == list(range(wl.seq_len))
        return 0, 0
    return selection_mismatch(gidx, ref["idx"], ref["pooled"], n, wl.window)


def assert_decode_close(got, ref):
    """Decode outputs against the oracle: the acceptance bar and the kernel's
    precision bound."""
    err = float(np.abs(np.asarray(got, np.float64) - ref).max()) if np.size(ref) else 0.0
    assert err <= DECODE_ATOL, f"max-abs error {err} above the acceptance bar {DECODE_ATOL}"
    assert err <= DECODE_PREC_ATOL, f"max-abs error {err} above the kernel precision bound"
    return err
