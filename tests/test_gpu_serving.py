"""The per-layer serving loop (Sec. 4.1; the decode shape of Table 3): every
layer calls ripple_decode_attn on its own compressed cache between stand-in
projections (plain torch matmuls on a hidden state; not the method), one
decode step of all layers captured in a CUDA graph and replayed per token.
Every step's attention outputs of every layer match the oracle's decode over
the grown caches, and the appended rows are the projected key/value rows."""
import numpy as np
import pytest
import torch

from oracle import ripple_oracle as O
from paper_2608_08684_gb300 import synth
from paper_2608_08684_gb300.serving import LayerDecodeLoop
from tests import gpu_common as C

pytestmark = pytest.mark.gpu
DEV = "cuda"


class StandIn:
    """Random per-layer projections hidden -> (q, k, v) and attention output ->
    hidden (residual), with per-layer buffers so that a step's rows can be read
    back after the graph has run."""

    def __init__(self, wl, seed):
        g = torch.Generator(device=DEV)
        g.manual_seed(seed)
        L, B, Hq, Hkv, d = wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim
        hid = Hq * d
        dt = wl.torch_dtype
        self.wl = wl
        self.h = torch.randn(B, hid, generator=g, device=DEV).to(dt)
        self.wqkv = [(torch.randn(hid, (Hq + 2 * Hkv) * d, generator=g, device=DEV)
                      / hid ** 0.5).to(dt) for _ in range(L)]
        self.wo = [(torch.randn(hid, hid, generator=g, device=DEV) / hid ** 0.5).to(dt)
                   for _ in range(L)]
        self.q = [torch.empty(1, B, Hq, d, dtype=dt, device=DEV) for _ in range(L)]
        self.k = [torch.empty(1, B, Hkv, d, dtype=dt, device=DEV) for _ in range(L)]
        self.v = [torch.empty(1, B, Hkv, d, dtype=dt, device=DEV) for _ in range(L)]

    def before(self, l):
        wl = self.wl
        B, Hq, Hkv, d = wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim
        # RMS-normalised hidden state, as a transformer layer's input: the
        # rows stay of unit scale however the residual stream grows
        hn = self.h.float()
        hn = (hn * torch.rsqrt(hn.square().mean(-1, keepdim=True) + 1e-6)).to(self.h.dtype)
        x = hn @ self.wqkv[l]
        self.q[l].copy_(x[:, :Hq * d].reshape(1, B, Hq, d))
        self.k[l].copy_(x[:, Hq * d:(Hq + Hkv) * d].reshape(1, B, Hkv, d))
        self.v[l].copy_(x[:, (Hq + Hkv) * d:].reshape(1, B, Hkv, d))
        return self.q[l], self.k[l], self.v[l]

    def after(self, l, out):
        wl = self.wl
        self.h.add_(out.reshape(wl.batch, -1).to(self.h.dtype) @ self.wo[l])


def _run(lib, wl, k_caches, v_caches, lens0, steps, seed):
    G, scale = wl.group, 1.0 / np.sqrt(wl.head_dim)
    rows_k = [[[synth.to_f64(k_caches[l][b, h, :lens0[l]]) for h in range(wl.n_kv_heads)]
               for b in range(wl.batch)] for l in range(wl.n_layers)]
    rows_v = [[[synth.to_f64(v_caches[l][b, h, :lens0[l]]) for h in range(wl.n_kv_heads)]
               for b in range(wl.batch)] for l in range(wl.n_layers)]
    lens = torch.tensor(lens0, dtype=torch.int32, device=DEV)
    sm = StandIn(wl, seed)
    loop = LayerDecodeLoop(k_caches, v_caches, lens, wl.n_q_heads, sm.before, sm.after)

    def check(t):
        # the oracle over the caches grown by this step's projected rows
        for l in range(wl.n_layers):
            q, kn, vn = (x[l][0].cpu() for x in (sm.q, sm.k, sm.v))
            got = loop.out[l][0].cpu().numpy()
            for b in range(wl.batch):
                for h in range(wl.n_kv_heads):
                    rows_k[l][b][h] = np.vstack([rows_k[l][b][h], synth.to_f64(kn[b, h])[None]])
                    rows_v[l][b][h] = np.vstack([rows_v[l][b][h], synth.to_f64(vn[b, h])[None]])
                    ref = O.decode_attention(synth.to_f64(q[b, h * G:(h + 1) * G]),
                                             rows_k[l][b][h], rows_v[l][b][h], scale)
                    C.assert_decode_close(got[b, h * G:(h + 1) * G], ref)
            # the appended rows are the projected rows, bit for bit
            assert torch.equal(k_caches[l][:, :, lens0[l] + t], sm.k[l][0])
            assert torch.equal(v_caches[l][:, :, lens0[l] + t], sm.v[l][0])

    loop.issue_step()  # eager first step (outside any capture)
    torch.cuda.synchronize()
    check(0)
    loop.capture()
    for t in range(1, steps):
        loop.replay()
        torch.cuda.synchronize()
        assert int(loop.status.item()) == 0
        check(t)
    assert lens.cpu().tolist() == [n + steps for n in lens0]


def test_serving_loop_tiny_after_compression(lib):
    # the tiny workload end to end: allocator budgets, compression of every
    # layer, then the per-layer loop
    wl = synth.WORKLOADS["tiny"]
    budgets = lib.ripple_alloc_budgets(synth.sensitivity_profile(wl), wl.ratio, wl.gamma,
                                       wl.global_budget)
    steps = 4
    k_caches, v_caches, lens0 = [], [], []
    for layer in range(wl.n_layers):
        q_win, k, v = (t.to(DEV) for t in C.layer_inputs(wl, layer, "cpu"))
        out = C.run_compress(lib, wl, budgets[layer], q_win, k, v, cap_extra=steps, scores=False)
        assert int(out["status"].item()) == 0
        k_caches.append(out["k_out"])
        v_caches.append(out["v_out"])
        lens0.append(out["n"])
    _run(lib, wl, k_caches, v_caches, lens0, steps, seed=5)


def test_serving_loop_llama8b_8k(lib):
    # the 8k Llama-3-8B-shaped stack (32 layers, bf16): caches at the RippleKV
    # sizes of its budgets, three steps through the captured graph
    wl = synth.WORKLOADS["llama8b-8k"]
    budgets = lib.ripple_alloc_budgets(synth.sensitivity_profile(wl), wl.ratio, wl.gamma,
                                       wl.global_budget)
    lens0 = [lib.ripple_keep_count(b, wl.seq_len, wl.window) for b in budgets]
    steps = 3
    kc, vc = zip(*[synth.decode_caches(wl, l, lens0[l] + steps, DEV) for l in range(wl.n_layers)])
    _run(lib, wl, list(kc), list(vc), lens0, steps, seed=6)
