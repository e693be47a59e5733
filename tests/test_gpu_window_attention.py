"""The scoring fused into the prefill attention of the observation-window rows
(ripple_compress_layers_attn): every layer's window-row attention output
against the oracle's causal softmax attention of those rows; its compression
against the oracle's (selection within the score tolerance of the threshold,
kept rows byte-exact), and bit for bit equal to ripple_compress_layers where
both split a unit's keys the same way (one item per unit).

Tolerance, from the kernel's arithmetic: the probabilities are final fp32
values (pass 1 fixed every row's normaliser) rounded once to bf16 for the
tensor cores, a relative error of at most 2^-8 each, so a row's output is off
by at most 2^-8 * sum_t p_t |v_t| (the oracle's own attention over |v|); the
fp32 accumulation, the exponentials (relative error ~2^-22) and the fp32 row
normalisers add far less: |gpu - oracle| <= 2^-8 * (p . |v|) + 2e-5 per
element."""
import numpy as np
import pytest
import torch

from oracle import ripple_oracle as O
from paper_2608_08684_gb300 import synth
from tests import gpu_common as C

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _run(lib, wl, budgets, attn=True):
    L = len(budgets)
    desc = lib.layer_desc(wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.seq_len,
                          wl.window, wl.pool_kernel, "max", wl.torch_dtype)
    B, H, d = wl.batch, wl.n_kv_heads, wl.head_dim
    ins = [tuple(t.to(DEV) for t in C.layer_inputs(wl, l, "cpu")) for l in range(L)]
    ns = [lib.ripple_keep_count(b, wl.seq_len, wl.window) for b in budgets]
    k_out = [torch.zeros(B, H, n + 2, d, dtype=wl.torch_dtype, device=DEV) for n in ns]
    v_out = [torch.zeros_like(x) for x in k_out]
    idx = [torch.full((B * H * n,), -1, dtype=torch.int32, device=DEV) for n in ns]
    tables = lib.CompressTables([x[0] for x in ins], [x[1] for x in ins], [x[2] for x in ins],
                                k_out, v_out, idx)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    o_win = None
    if attn:
        o_win = [torch.full((B, wl.n_q_heads, wl.window, d), float("nan"), device=DEV)
                 for _ in range(L)]
        ws = torch.empty(lib.ripple_compress_layers_attn_workspace_bytes(desc, L),
                         dtype=torch.uint8, device=DEV)
        got = lib.ripple_compress_layers_attn(desc, budgets, tables, o_win, ws, dev_status=status)
    else:
        ws = torch.empty(lib.ripple_compress_layers_workspace_bytes(desc, L), dtype=torch.uint8,
                         device=DEV)
        got = lib.ripple_compress_layers(desc, budgets, tables, ws, dev_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert got == ns
    return dict(ins=ins, idx=idx, k_out=k_out, v_out=v_out, o_win=o_win, n=ns)


def _check_compression(wl, res, budgets, units=None):
    """Every (or the listed) unit's retained set against the oracle's."""
    B, H = wl.batch, wl.n_kv_heads
    agree = total = 0
    for l, (q, k, v) in enumerate(res["ins"]):
        n = res["n"][l]
        out = {"n": n, "idx": res["idx"][l].view(B, H, n), "k_out": res["k_out"][l],
               "v_out": res["v_out"][l], "scores": None}
        for b in range(B):
            for h in range(H):
                if units is not None and (b, h) not in units:
                    continue
                a, t = C.check_compress_unit(wl, out, q, k, v, b, h, budgets[l])
                agree, total = agree + a, total + t
    assert agree >= 0.999 * total, (agree, total)


def _check_outputs(wl, res, units=None):
    G, scale = wl.group, 1.0 / np.sqrt(wl.head_dim)
    for l, (q, k, v) in enumerate(res["ins"]):
        o = res["o_win"][l].cpu().numpy()
        assert np.isfinite(o).all()
        for b in range(wl.batch):
            for h in range(wl.n_kv_heads):
                if units is not None and (b, h) not in units:
                    continue
                qq, kk, vv = C.unit_f64(wl, q, k, v, b, h)
                ref = O.window_attention(qq, kk, vv, scale)
                bound = 2.0 ** -8 * O.window_attention(qq, kk, np.abs(vv), scale) + 2e-5
                err = np.abs(o[b, h * G:(h + 1) * G] - ref)
                assert np.all(err <= bound), (l, b, h, float(err.max()), float((err - bound).max()))


SHAPES = [
    # G * w = 128: G 4, w 32; ragged last tile, window keys inside it
    ("G4-T1000", dict(n_layers=2, batch=2, n_q_heads=8, n_kv_heads=2, head_dim=128, seq_len=1000,
                      dtype="bf16", kv_dist="scaled_sinks", seed=81), [31, 400]),
    # window keys across two tiles (P = 100), a single-tile prefix
    ("G4-T132", dict(n_layers=1, batch=1, n_q_heads=4, n_kv_heads=1, head_dim=128, seq_len=132,
                     dtype="bf16", seed=82), [60]),
    # two items per unit (the partial outputs summed in item order)
    ("G4-T33000", dict(n_layers=2, batch=1, n_q_heads=8, n_kv_heads=2, head_dim=128,
                       seq_len=33000, dtype="bf16", kv_dist="scaled_sinks", seed=83),
     [700, 10**6]),
    # G 8, w 16
    ("G8-w16", dict(n_layers=2, batch=1, n_q_heads=16, n_kv_heads=2, head_dim=128, seq_len=777,
                    window=16, dtype="bf16", seed=84), [100, 50]),
]


@pytest.mark.parametrize("name,over,budgets", SHAPES, ids=[s[0] for s in SHAPES])
def test_window_attention_matches_oracle(lib, name, over, budgets):
    wl = synth.WORKLOADS["tiny"].replace(**over)
    res = _run(lib, wl, budgets)
    _check_outputs(wl, res)
    _check_compression(wl, res, budgets)
    if -(-wl.seq_len // 128) <= 9:
        # one item per unit in both calls: the compression equals
        # ripple_compress_layers' bit for bit
        ref = _run(lib, wl, budgets, attn=False)
        for key in ("idx", "k_out", "v_out"):
            for x, y in zip(res[key], ref[key]):
                assert torch.equal(x, y), (name, key)


def test_window_attention_full_size_sampled(lib):
    # the 32k Llama-3-8B-shaped layer: 4 layers in one call, 2 units checked
    wl = synth.WORKLOADS["llama8b-32k"].replace(n_layers=4)
    budgets = [1024, 3000, 500, 10**7]
    res = _run(lib, wl, budgets)
    units = {(0, 0), (wl.batch - 1, wl.n_kv_heads - 1)}
    _check_outputs(wl, res, units=units)
    _check_compression(wl, res, budgets, units=units)


def test_window_attention_is_reproducible(lib):
    wl = synth.WORKLOADS["tiny"].replace(**SHAPES[2][1])
    a = _run(lib, wl, SHAPES[2][2])
    b = _run(lib, wl, SHAPES[2][2])
    for x, y in zip(a["o_win"], b["o_win"]):
        assert torch.equal(x, y)


def test_window_attention_rejects_other_shapes(lib):
    wl = synth.WORKLOADS["tiny"].replace(n_layers=1, batch=1, n_q_heads=16, n_kv_heads=2,
                                         head_dim=128, seq_len=300, dtype="bf16")  # G * w = 256
    desc = lib.layer_desc(wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.seq_len,
                          wl.window, wl.pool_kernel, "max", wl.torch_dtype)
    with pytest.raises(lib.RippleError):
        lib.ripple_compress_layers_attn_workspace_bytes(desc, 1)
