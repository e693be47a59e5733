"""Parity of the profiling kernels (Sec. 4.3) with the CPU oracle on the same
seeded inputs, through the C ABI: the Value perturbation of Eq. 6 and the
window KL divergence of Eq. 7.

Tolerances, from the fp32 arithmetic of the kernels:
* perturbation, fp32 caches: the squared norm is a sum of d squares (four per
  lane, then a shuffle tree), the square root and alpha * norm add a few
  roundings and the final fused multiply-add one more: within 2^-20 of
  |v| + alpha ||v|| |eps| per element. bf16 caches: the fp32 result is rounded
  once to bf16, so it equals the fp64 result rounded to bf16 except where the
  fp64 value lies within that fp32 bound of a rounding midpoint, where the
  two are adjacent bf16 values.
* window KL: shares of 512 logits reduced in fp32 (weights from the
  special-function exponential, relative error about 2^-22 each; 32-term
  thread sums and shuffle trees), rows merged in double. Where every share
  stays in the Taylor regime (|x| <= 1/2) the divergence is formed as
  log1p(E[x] + E[g(x)]) - E[x]: the weights and the positive sum of g carry
  relative errors of about 1e-6, and the error of E[x] enters only times
  E[x] itself, so the error is relative to the divergence:
  |gpu - oracle| <= 1e-4 |oracle| + 1e-10 at divergences of 1e-5 to 1e-4.
  Elsewhere the shares' masses are summed in the log domain with relative
  errors of about 1e-6, which reach the divergence as absolute errors of a
  few 1e-7 to 1e-6: |gpu - oracle| <= 1e-3 |oracle| + 2e-5.
"""
import math

import numpy as np
import pytest
import torch

from oracle import ripple_oracle as O
from paper_2608_08684_gb300 import synth

pytestmark = pytest.mark.gpu
DEV = "cuda"
PERTURB_F32_REL = 2.0 ** -20
KL_RTOL, KL_ATOL = 1e-3, 2e-5
KL_SMALL_RTOL, KL_SMALL_ATOL = 1e-4, 1e-10


def _perturb_case(lib, B, H, T, d, dtype, pb, pe, in_place, alpha, seed):
    wl = synth.WORKLOADS["tiny"].replace(batch=B, n_kv_heads=H, n_q_heads=H, seq_len=T,
                                         head_dim=d, dtype=dtype, seed=seed, window=1)
    v = synth.layer_values(wl, 0, DEV)
    # rows of very different norms: scale each row by a lognormal factor
    g = torch.Generator(device=DEV)
    g.manual_seed(seed)
    scale = torch.exp(torch.randn(B, H, T, 1, generator=g, device=DEV))
    v = (v.float() * scale).to(v.dtype).contiguous()
    eps = synth.perturb_draws(wl, 0, pe - pb, DEV).contiguous()
    v_in = v.clone()
    if in_place:
        lib.ripple_perturb_values(v, eps if pe > pb else None, alpha, pb, pe)
        out = v
    else:
        out = torch.full_like(v, float("nan"))
        lib.ripple_perturb_values(v, eps if pe > pb else None, alpha, pb, pe, v_out=out)
    torch.cuda.synchronize()
    return v_in, eps, out


def _check_perturbed(v_in, eps, out, alpha, pb, pe):
    alpha32 = float(np.float32(alpha))  # the kernel's alpha is fp32
    vv = synth.to_f64(v_in)
    ee = synth.to_f64(eps)
    want = O.perturb_values(vv, ee, alpha32, pb, pe)
    got = synth.to_f64(out)
    # protected rows: bit-exact copies (or untouched in place)
    assert torch.equal(out[:, :, :pb], v_in[:, :, :pb])
    assert torch.equal(out[:, :, pe:], v_in[:, :, pe:])
    if pe == pb:
        return
    rows = vv[:, :, pb:pe]
    bound = PERTURB_F32_REL * (np.abs(rows) + alpha32 * np.linalg.norm(rows, axis=-1,
                                                                       keepdims=True)
                               * np.abs(ee))
    w = want[:, :, pb:pe]
    gr = got[:, :, pb:pe]
    if out.dtype == torch.float32:
        err = np.abs(gr - w)
        assert np.all(err <= bound + 2.0 ** -24 * np.abs(w)), err.max()
    else:
        w16 = synth.to_f64(torch.from_numpy(w).to(torch.bfloat16))
        diff = gr != w16
        if diff.any():
            # only where the fp64 value sits within the fp32 error of a midpoint
            mid = (gr[diff] + w16[diff]) / 2.0
            assert np.all(np.abs(w[diff] - mid) <= bound[diff]), np.abs(w[diff] - mid).max()
            ulp = np.abs(gr[diff] - w16[diff])
            assert np.all(ulp <= 2.0 ** (np.floor(np.log2(np.abs(w[diff]))) - 6))
        assert diff.mean() < 0.01


@pytest.mark.parametrize("B,H,T,d,dtype,pb,pe,in_place", [
    (2, 3, 300, 128, "bf16", 0, 268, False),
    (1, 8, 1000, 128, "bf16", 17, 968, True),
    (2, 2, 513, 64, "f32", 5, 500, False),
    (1, 3, 77, 64, "bf16", 0, 77, True),
    (3, 1, 129, 128, "f32", 1, 128, True),
    (2, 2, 100, 128, "bf16", 40, 40, False),
    (2, 2, 100, 64, "f32", 40, 40, True),
], ids=["bf16-d128-window", "bf16-d128-inplace", "f32-d64", "bf16-d64-all-inplace",
        "f32-d128-inplace", "empty-range-copy", "empty-range-inplace"])
def test_perturbation_matches_oracle(lib, B, H, T, d, dtype, pb, pe, in_place):
    v_in, eps, out = _perturb_case(lib, B, H, T, d, dtype, pb, pe, in_place, 0.1, seed=71 + T)
    _check_perturbed(v_in, eps, out, 0.1, pb, pe)


def test_perturbation_full_size_layer_sampled(lib):
    # the benchmark's shape: one Llama-3-8B-sized layer at 32k, B = 4, bf16,
    # the 32-token observation window protected; rows checked on a sample
    wl = synth.WORKLOADS["llama8b-32k"]
    B, H, T, d = wl.batch, wl.n_kv_heads, wl.seq_len, wl.head_dim
    pb, pe, alpha = 0, T - wl.window, 0.05
    v = synth.layer_values(wl, 3, DEV)
    eps = synth.perturb_draws(wl, 3, pe - pb, DEV)
    out = torch.empty_like(v)
    lib.ripple_perturb_values(v, eps, alpha, pb, pe, v_out=out)
    torch.cuda.synchronize()
    assert torch.equal(out[:, :, pe:], v[:, :, pe:])
    g = torch.Generator()
    g.manual_seed(5)
    for _ in range(6):
        b, h = int(torch.randint(0, B, (1,), generator=g)), int(torch.randint(0, H, (1,), generator=g))
        u0 = int(torch.randint(0, pe - 64, (1,), generator=g))
        sl = slice(u0, u0 + 64)
        _check_perturbed(v[b:b + 1, h:h + 1, sl], eps[b:b + 1, h:h + 1, sl],
                         out[b:b + 1, h:h + 1, sl], alpha, 0, 64)


def test_perturbation_alpha_zero_is_a_copy(lib):
    wl = synth.WORKLOADS["tiny"].replace(batch=2, n_kv_heads=2, n_q_heads=2, seq_len=64,
                                         head_dim=128, dtype="bf16", window=1)
    v = synth.layer_values(wl, 0, DEV)
    eps = synth.perturb_draws(wl, 0, 60, DEV)
    out = torch.empty_like(v)
    lib.ripple_perturb_values(v, eps, 0.0, 2, 62, v_out=out)
    torch.cuda.synchronize()
    assert torch.equal(out, v)


def _kl_check(got, want):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    err = np.abs(got - want)
    assert np.all(err <= KL_RTOL * np.abs(want) + KL_ATOL), (err.max(), got, want)


@pytest.mark.parametrize("n_sets,n_pos,vocab,dtype", [
    (3, 5, 128256, torch.float32),
    (2, 4, 32768, torch.bfloat16),
    (2, 3, 8, torch.float32),
    (2, 2, 8200, torch.bfloat16),
    (1, 300, 1000, torch.float32),
], ids=["f32-llama3-vocab", "bf16-mistral-vocab", "vocab8", "two-slices-ragged",
        "300-positions"])
def test_window_kl_matches_oracle(lib, n_sets, n_pos, vocab, dtype):
    p, q = synth.window_logits(90 + vocab % 97, n_sets, n_pos, vocab, dtype, DEV)
    ws = torch.empty(lib.ripple_window_kl_workspace_bytes(n_sets, n_pos, vocab),
                     dtype=torch.uint8, device=DEV)
    d_out = torch.full((n_sets,), float("nan"), device=DEV)
    kl_out = torch.full((n_sets, n_pos), float("nan"), device=DEV)
    lib.ripple_window_kl(p, q, ws, d_out, kl_out)
    torch.cuda.synchronize()
    pp = synth.to_f64(p)
    for s in range(n_sets):
        kl, d = O.window_kl(pp, synth.to_f64(q[s]))
        _kl_check(kl_out[s].cpu().numpy(), kl)
        _kl_check([d_out[s].item()], [d])


def test_window_kl_identical_rows_give_exact_zero_and_shift_near_zero(lib):
    n_pos, vocab = 6, 50000
    p, q = synth.window_logits(7, 3, n_pos, vocab, torch.float32, DEV)
    q[0] = p          # identical run
    q[1] = p + 37.25  # constant shift: same distribution
    ws = torch.empty(lib.ripple_window_kl_workspace_bytes(3, n_pos, vocab), dtype=torch.uint8,
                     device=DEV)
    d_out = torch.empty(3, device=DEV)
    kl_out = torch.empty(3, n_pos, device=DEV)
    lib.ripple_window_kl(p, q, ws, d_out, kl_out)
    torch.cuda.synchronize()
    assert torch.all(kl_out[0] == 0) and d_out[0].item() == 0.0
    assert torch.all(kl_out[1].abs() <= KL_ATOL)
    kl, d = O.window_kl(synth.to_f64(p), synth.to_f64(q[2]))
    _kl_check(kl_out[2].cpu().numpy(), kl)


def test_window_kl_large_perturbation_and_without_per_position_output(lib):
    # a set whose perturbation reshapes the distribution (sigma 3: KL of order one)
    n_pos, vocab = 4, 20000
    p, q = synth.window_logits(8, 2, n_pos, vocab, torch.float32, DEV, sigmas=[3.0, 0.01])
    ws = torch.empty(lib.ripple_window_kl_workspace_bytes(2, n_pos, vocab), dtype=torch.uint8,
                     device=DEV)
    d_out = torch.empty(2, device=DEV)
    lib.ripple_window_kl(p, q, ws, d_out)
    torch.cuda.synchronize()
    for s in range(2):
        _, d = O.window_kl(synth.to_f64(p), synth.to_f64(q[s]))
        _kl_check([d_out[s].item()], [d])
    assert d_out[0].item() > 1.0 > 1e-3 > d_out[1].item() > 0


def test_window_kl_small_divergence_keeps_relative_precision(lib):
    # perturbations of sigma 0.014 and 0.004: divergences near 1e-4 and 1e-5,
    # every share in the Taylor regime
    n_pos, vocab = 8, 128256
    for dtype in (torch.float32, torch.bfloat16):
        p, q = synth.window_logits(31, 2, n_pos, vocab, dtype, DEV, sigmas=[0.014, 0.004])
        ws = torch.empty(lib.ripple_window_kl_workspace_bytes(2, n_pos, vocab),
                         dtype=torch.uint8, device=DEV)
        d_out = torch.empty(2, device=DEV)
        kl_out = torch.empty(2, n_pos, device=DEV)
        lib.ripple_window_kl(p, q, ws, d_out, kl_out)
        torch.cuda.synchronize()
        pp = synth.to_f64(p)
        for s in range(2):
            kl, d = O.window_kl(pp, synth.to_f64(q[s]))
            if dtype == torch.float32:
                assert 1e-6 < kl.min() and kl.max() < 3e-4
            got = np.concatenate([kl_out[s].cpu().numpy().astype(np.float64), [d_out[s].item()]])
            want = np.concatenate([kl, [d]])
            err = np.abs(got - want)
            assert np.all(err <= KL_SMALL_RTOL * np.abs(want) + KL_SMALL_ATOL), \
                (dtype, s, (err / np.abs(want)).max())


def test_window_kl_far_logits_and_shifts(lib):
    n_pos, vocab = 5, 40000
    p, q = synth.window_logits(32, 4, n_pos, vocab, torch.float32, DEV,
                               sigmas=[0.01, 0.01, 0.01, 0.01])
    q[0, :, 17] += 6.0      # two far logits: their shares leave the Taylor regime
    q[0, :, 30001] -= 9.0
    q[1, :, 123] += 120.0   # exp(q - q at the largest p) overflows fp32 in that share
    q[2] = p - 100.0        # constant shift: the same distribution
    q[3, :, 8191] += 0.75   # one far logit at a slice's last entry
    ws = torch.empty(lib.ripple_window_kl_workspace_bytes(4, n_pos, vocab), dtype=torch.uint8,
                     device=DEV)
    d_out = torch.empty(4, device=DEV)
    kl_out = torch.empty(4, n_pos, device=DEV)
    lib.ripple_window_kl(p, q, ws, d_out, kl_out)
    torch.cuda.synchronize()
    pp = synth.to_f64(p)
    for s in range(4):
        kl, d = O.window_kl(pp, synth.to_f64(q[s]))
        _kl_check(kl_out[s].cpu().numpy(), kl)
        _kl_check([d_out[s].item()], [d])
    assert d_out[1].item() > 50.0 and abs(d_out[2].item()) <= KL_ATOL


def test_window_kl_workspace_contents_and_graph_replay(lib):
    n_sets, n_pos, vocab = 3, 7, 20000
    p, q = synth.window_logits(33, n_sets, n_pos, vocab, torch.float32, DEV)
    nbytes = lib.ripple_window_kl_workspace_bytes(n_sets, n_pos, vocab)
    ref_kl = torch.empty(n_sets, n_pos, device=DEV)
    ref_d = torch.empty(n_sets, device=DEV)
    lib.ripple_window_kl(p, q, torch.zeros(nbytes, dtype=torch.uint8, device=DEV), ref_d, ref_kl)
    # arbitrary workspace contents (every counter word 0xA5A5A5A5)
    ws = torch.full((nbytes,), 0xA5, dtype=torch.uint8, device=DEV)
    kl_out = torch.full((n_sets, n_pos), float("nan"), device=DEV)
    d_out = torch.full((n_sets,), float("nan"), device=DEV)
    lib.ripple_window_kl(p, q, ws, d_out, kl_out)
    torch.cuda.synchronize()
    assert torch.equal(kl_out, ref_kl) and torch.equal(d_out, ref_d)
    # one call captured in a CUDA graph, replayed twice
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        lib.ripple_window_kl(p, q, ws, d_out, kl_out)
    for _ in range(2):
        kl_out.fill_(float("nan"))
        d_out.fill_(float("nan"))
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(kl_out, ref_kl) and torch.equal(d_out, ref_d)


def test_window_kl_is_reproducible(lib):
    p, q = synth.window_logits(9, 4, 8, 128256, torch.bfloat16, DEV)
    ws = torch.empty(lib.ripple_window_kl_workspace_bytes(4, 8, 128256), dtype=torch.uint8,
                     device=DEV)
    outs = []
    for _ in range(2):
        kl_out = torch.empty(4, 8, device=DEV)
        d_out = torch.empty(4, device=DEV)
        lib.ripple_window_kl(p, q, ws, d_out, kl_out)
        outs.append((kl_out.clone(), d_out.clone()))
    torch.cuda.synchronize()
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_profile_chain_feeds_the_allocator(lib):
    # Algorithm 1's profiling half on stand-in outputs: per example, the window
    # KL of every layer's perturbed run (GPU), then Eq. 8 and Eqs. 9-12 (host C);
    # the allocator's input equals the oracle's average of the GPU responses.
    L, N, n_pos, vocab = 6, 3, 8, 4096
    ws = torch.empty(lib.ripple_window_kl_workspace_bytes(L, n_pos, vocab), dtype=torch.uint8,
                     device=DEV)
    d = []
    for i in range(N):
        sig = [0.05 + 0.3 * math.exp(-((l - 2.5) ** 2) / 2.0) for l in range(L)]
        p, q = synth.window_logits(200 + i, L, n_pos, vocab, torch.float32, DEV, sigmas=sig)
        d_out = torch.empty(L, device=DEV)
        lib.ripple_window_kl(p, q, ws, d_out)
        d.append([float(x) for x in d_out.cpu()])
        for l in (0, 3):
            _, want = O.window_kl(synth.to_f64(p), synth.to_f64(q[l]))
            _kl_check([d[-1][l]], [want])
    s = lib.ripple_sensitivity_profile(d)
    assert s == [float(x) for x in O.sensitivity_profile(d)]
    budgets = lib.ripple_alloc_budgets(s, 1.5, 0.0, 1024 * L)
    assert budgets == O.alloc_budgets(s, 1.5, 0.0, 1024 * L)
    assert sum(budgets) == 1024 * L and max(budgets) == budgets[int(np.argmax(s))]
