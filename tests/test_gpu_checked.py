"""The bounds-checked build (libripple_checked.so, RIPPLE_CHECKED): every
guarded global access of the kernels tests its offset against its buffer's
extent and would report RIPPLE_EBOUNDS in the status word instead of going
out of bounds. It stands in for a memory checker, which is not available on
these GPUs. Both builds are loaded side by side (a second instance of the
binding over the checked library). On shapes that exercise every scoring path
(tensor cores with 128 and 256 window rows, fp32 on the CUDA cores), the
three selection kernels, the gather, split and single decode items in both
dtypes, the no-allocation decode and the window divergence with ragged
slices and empty shares, the checked build reports no violation and its
outputs equal the normal build's bit for bit (the guards change no
arithmetic when an access is in bounds)."""
import importlib.util
import os

import pytest
import torch

from paper_2608_08684_gb300 import synth
from tests import gpu_common as C

pytestmark = pytest.mark.gpu
DEV = "cuda"
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def chk():
    """A second instance of the binding, over the checked library."""
    from paper_2608_08684_gb300 import build as _build
    _build.build_library(checked=True)
    path = os.path.join(ROOT, "paper_2608_08684_gb300", "ripple.py")
    old = os.environ.get("RIPPLE_CHECKED")
    os.environ["RIPPLE_CHECKED"] = "1"
    try:
        spec = importlib.util.spec_from_file_location("ripple_checked_binding", path)
        mod = importlib.util.module_from_spec(spec)
        spec.loader.exec_module(mod)
    finally:
        if old is None:
            del os.environ["RIPPLE_CHECKED"]
        else:
            os.environ["RIPPLE_CHECKED"] = old
    assert mod.CHECKED and mod.LIB_PATH.endswith("libripple_checked.so")
    return mod


COMPRESS = [
    # 128 window rows: tcgen05 scoring, cluster selection (few units)
    ("tc-128", dict(batch=2, n_q_heads=8, n_kv_heads=2, head_dim=128, seq_len=1000, dtype="bf16",
                    kv_dist="scaled_sinks", seed=61), [31, 200, 968, 10**6]),
    # 256 window rows: the other tcgen05 kernel
    ("tc-256", dict(batch=1, n_q_heads=16, n_kv_heads=2, head_dim=128, seq_len=700, dtype="bf16",
                    seed=62), [50, 300]),
    # fp32, d = 64: scoring on the CUDA cores
    ("simt-f32", dict(batch=1, n_q_heads=4, n_kv_heads=2, head_dim=64, seq_len=389, dtype="f32",
                      seed=63), [10, 128]),
]


@pytest.mark.parametrize("name,over,budgets", COMPRESS, ids=[c[0] for c in COMPRESS])
def test_compress_layer_checked(lib, chk, name, over, budgets):
    wl = synth.WORKLOADS["tiny"].replace(**over)
    q_win, k, v = (t.to(DEV) for t in C.layer_inputs(wl, 0, "cpu"))
    for budget in budgets:
        a = C.run_compress(lib, wl, budget, q_win, k, v, cap_extra=2)
        b = C.run_compress(chk, wl, budget, q_win, k, v, cap_extra=2)
        assert int(b["status"].item()) == 0, (name, budget, int(b["status"].item()))
        for key in ("idx", "k_out", "v_out", "scores"):
            assert torch.equal(a[key], b[key]), (name, budget, key)


def test_compress_layers_checked(lib, chk):
    # 32 layers x 8 units: one 1024-thread selection CTA per unit
    wl = synth.WORKLOADS["tiny"].replace(n_layers=32, batch=1, n_q_heads=32, n_kv_heads=8,
                                         head_dim=128, seq_len=640, dtype="bf16", seed=64)
    budgets = [32 + 19 * l for l in range(wl.n_layers)]
    B, H, d = wl.batch, wl.n_kv_heads, wl.head_dim
    ins = [tuple(t.to(DEV) for t in C.layer_inputs(wl, l, "cpu")) for l in range(wl.n_layers)]
    results = []
    for m in (lib, chk):
        desc = m.layer_desc(B, wl.n_q_heads, H, d, wl.seq_len, wl.window, wl.pool_kernel, "max",
                            wl.torch_dtype)
        ns = [m.ripple_keep_count(x, wl.seq_len, wl.window) for x in budgets]
        k_out = [torch.zeros(B, H, n + 2, d, dtype=wl.torch_dtype, device=DEV) for n in ns]
        v_out = [torch.zeros_like(x) for x in k_out]
        idx = [torch.full((B * H * n,), -1, dtype=torch.int32, device=DEV) for n in ns]
        tables = m.CompressTables([x[0] for x in ins], [x[1] for x in ins], [x[2] for x in ins],
                                  k_out, v_out, idx)
        ws = torch.empty(m.ripple_compress_layers_workspace_bytes(desc, wl.n_layers),
                         dtype=torch.uint8, device=DEV)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        m.ripple_compress_layers(desc, budgets, tables, ws, dev_status=status)
        torch.cuda.synchronize()
        results.append((int(status.item()), idx, k_out, v_out))
    assert results[1][0] == 0
    for x, y in zip(results[0][1] + results[0][2] + results[0][3],
                    results[1][1] + results[1][2] + results[1][3]):
        assert torch.equal(x, y)


DECODE = [
    # groups split over several items (partials and their combine)
    ("split-G4", dict(n_layers=3, batch=1, n_q_heads=8, n_kv_heads=2, head_dim=128, dtype="bf16",
                      seed=65), [2047, 4097, 8300]),
    ("G8-f32", dict(n_layers=2, batch=2, n_q_heads=16, n_kv_heads=2, head_dim=64, dtype="f32",
                    seed=66), [0, 513]),
    ("G1-single-layer", dict(n_layers=1, batch=2, n_q_heads=2, n_kv_heads=2, head_dim=128,
                             dtype="bf16", seed=67), [3000]),
]


@pytest.mark.parametrize("name,over,lens0", DECODE, ids=[c[0] for c in DECODE])
def test_decode_checked(lib, chk, name, over, lens0):
    wl = synth.WORKLOADS["tiny"].replace(**over)
    caps = [n + 3 for n in lens0]
    base = [synth.decode_caches(wl, i, caps[i]) for i in range(wl.n_layers)]
    runs = []
    for m in (lib, chk):
        kc = [x[0].to(DEV) for x in base]
        vc = [x[1].to(DEV) for x in base]
        desc = m.decode_desc(wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim,
                             wl.torch_dtype)
        tables = m.DecodeTables(kc, vc)
        ws = torch.empty(m.ripple_decode_workspace_bytes(desc, caps), dtype=torch.uint8,
                         device=DEV)
        lens = torch.tensor(lens0, dtype=torch.int32, device=DEV)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        outs = []
        for step in range(2):
            q, kn, vn = (t.to(DEV) for t in synth.decode_inputs(wl, step))
            out = torch.empty(wl.n_layers, wl.batch, wl.n_q_heads, wl.head_dim, device=DEV)
            m.ripple_decode_attn(desc, q, kn, vn, tables, lens, out, ws, dev_status=status)
            outs.append(out)
        # the no-allocation entry point on the same caches, one more step
        q, kn, vn = (t.to(DEV) for t in synth.decode_inputs(wl, 2))
        out = torch.empty(wl.n_layers, wl.batch, wl.n_q_heads, wl.head_dim, device=DEV)
        m.ripple_decode_attn_noalloc(desc, q, kn, vn, tables, lens, out, dev_status=status)
        outs.append(out)
        torch.cuda.synchronize()
        runs.append((int(status.item()), outs, kc, vc, lens))
    assert runs[1][0] == 0, runs[1][0]
    for x, y in zip(runs[0][1] + runs[0][2] + runs[0][3] + [runs[0][4]],
                    runs[1][1] + runs[1][2] + runs[1][3] + [runs[1][4]]):
        assert torch.equal(x, y)


KL = [(2, 3, 8, torch.float32), (2, 2, 8200, torch.bfloat16), (3, 5, 40000, torch.float32)]


@pytest.mark.parametrize("n_sets,n_pos,vocab,dtype", KL)
def test_window_kl_checked(lib, chk, n_sets, n_pos, vocab, dtype):
    p, q = synth.window_logits(70 + vocab % 13, n_sets, n_pos, vocab, dtype, DEV)
    if vocab > 8192:
        q[0, :, 5] += 6.0  # a share outside the Taylor regime
    runs = []
    for m in (lib, chk):
        ws = torch.empty(m.ripple_window_kl_workspace_bytes(n_sets, n_pos, vocab),
                         dtype=torch.uint8, device=DEV)
        d_out = torch.empty(n_sets, device=DEV)
        kl_out = torch.empty(n_sets, n_pos, device=DEV)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        m.ripple_window_kl(p, q, ws, d_out, kl_out, dev_status=status)
        torch.cuda.synchronize()
        runs.append((int(status.item()), d_out, kl_out))
    assert runs[1][0] == 0
    assert torch.equal(runs[0][1], runs[1][1]) and torch.equal(runs[0][2], runs[1][2])


def test_compress_layers_attn_checked(lib, chk):
    # the scoring fused into the window rows' prefill attention (several items
    # per unit, window keys across the last tiles)
    wl = synth.WORKLOADS["tiny"].replace(n_layers=2, batch=1, n_q_heads=8, n_kv_heads=2,
                                         head_dim=128, seq_len=33000, dtype="bf16", seed=68)
    budgets = [300, 1500]
    B, H, d = wl.batch, wl.n_kv_heads, wl.head_dim
    ins = [tuple(t.to(DEV) for t in C.layer_inputs(wl, l, "cpu")) for l in range(wl.n_layers)]
    results = []
    for m in (lib, chk):
        desc = m.layer_desc(B, wl.n_q_heads, H, d, wl.seq_len, wl.window, wl.pool_kernel, "max",
                            wl.torch_dtype)
        ns = [m.ripple_keep_count(x, wl.seq_len, wl.window) for x in budgets]
        k_out = [torch.zeros(B, H, n, d, dtype=wl.torch_dtype, device=DEV) for n in ns]
        v_out = [torch.zeros_like(x) for x in k_out]
        idx = [torch.full((B * H * n,), -1, dtype=torch.int32, device=DEV) for n in ns]
        o_win = [torch.empty(B, wl.n_q_heads, wl.window, d, device=DEV) for _ in ns]
        tables = m.CompressTables([x[0] for x in ins], [x[1] for x in ins], [x[2] for x in ins],
                                  k_out, v_out, idx)
        ws = torch.empty(m.ripple_compress_layers_attn_workspace_bytes(desc, wl.n_layers),
                         dtype=torch.uint8, device=DEV)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        m.ripple_compress_layers_attn(desc, budgets, tables, o_win, ws, dev_status=status)
        torch.cuda.synchronize()
        results.append((int(status.item()), idx + k_out + v_out + o_win))
    assert results[1][0] == 0
    for x, y in zip(results[0][1], results[1][1]):
        assert torch.equal(x, y)
