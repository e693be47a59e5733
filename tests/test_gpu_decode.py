"""GPU parity of ragged GQA decode attention (ripple_decode_attn) against the
CPU oracle on seeded caches: outputs within 2e-2 max-abs of the fp64 oracle,
appended rows byte-exact, lengths advanced, full caches reported; and the
end-to-end compress -> decode path, including budget >= T reproducing full
attention exactly."""
import numpy as np
import pytest
import torch

from oracle import ripple_oracle as O
from paper_2608_08684_gb300 import synth
from tests import gpu_common as C

pytestmark = pytest.mark.gpu
DEV = "cuda"


class Session:
    """Caches, lengths and workspace of one multi-layer decode run."""

    def __init__(self, lib, wl, layers, caps, lens0, k_caches, v_caches):
        self.lib, self.wl, self.layers = lib, wl, list(layers)
        self.k = [t.to(DEV).contiguous() for t in k_caches]
        self.v = [t.to(DEV).contiguous() for t in v_caches]
        self.caps = list(caps)
        self.lens = torch.tensor(lens0, dtype=torch.int32, device=DEV)
        self.desc = lib.decode_desc(len(self.layers), wl.batch, wl.n_q_heads, wl.n_kv_heads,
                                    wl.head_dim, wl.torch_dtype)
        self.tables = lib.DecodeTables(self.k, self.v)
        self.ws = torch.empty(lib.ripple_decode_workspace_bytes(self.desc, self.caps),
                              dtype=torch.uint8, device=DEV)
        self.status = torch.zeros(1, dtype=torch.int32, device=DEV)
        self.out = torch.empty(len(self.layers), wl.batch, wl.n_q_heads, wl.head_dim,
                               dtype=torch.float32, device=DEV)

    def step(self, q, k_new, v_new):
        self.lib.ripple_decode_attn(self.desc, q.to(DEV), k_new.to(DEV), v_new.to(DEV),
                                    self.tables, self.lens, self.out, self.ws,
                                    dev_status=self.status)
        torch.cuda.synchronize()
        return self.out.cpu().numpy()


def _oracle_step(wl, rows_k, rows_v, q, k_new, v_new):
    """Oracle decode of every (layer, b, q head); rows_* lists are appended in place."""
    G = wl.group
    scale = 1.0 / np.sqrt(wl.head_dim)
    L = len(rows_k)
    out = np.zeros((L, wl.batch, wl.n_q_heads, wl.head_dim))
    for i in range(L):
        for b in range(wl.batch):
            for h in range(wl.n_kv_heads):
                rows_k[i][b][h] = np.vstack([rows_k[i][b][h], synth.to_f64(k_new[i, b, h])[None]])
                rows_v[i][b][h] = np.vstack([rows_v[i][b][h], synth.to_f64(v_new[i, b, h])[None]])
                qg = synth.to_f64(q[i, b, h * G:(h + 1) * G])
                out[i, b, h * G:(h + 1) * G] = O.decode_attention(qg, rows_k[i][b][h],
                                                                  rows_v[i][b][h], scale)
    return out


DECODE_SHAPES = [
    ("tiny-f32", dict(), [5, 130, 257, 0]),
    ("bf16-d128-G4", dict(n_layers=3, batch=2, n_q_heads=8, n_kv_heads=2, head_dim=128,
                          dtype="bf16", kv_dist="scaled_sinks", seed=41), [1, 128, 300]),
    ("bf16-d128-G8", dict(n_layers=2, batch=1, n_q_heads=16, n_kv_heads=2, head_dim=128,
                          dtype="bf16", seed=42), [127, 513]),
    ("bf16-d64-G1", dict(n_layers=2, batch=2, n_q_heads=3, n_kv_heads=3, head_dim=64,
                         dtype="bf16", seed=43), [64, 200]),
    # groups split over several work items, item edges and a ragged tail: with
    # few groups the items shrink to 256 rows (fewer items than SMs otherwise)
    ("bf16-d128-G4-split", dict(n_layers=4, batch=1, n_q_heads=8, n_kv_heads=2, head_dim=128,
                                dtype="bf16", kv_dist="scaled_sinks", seed=47),
     [2047, 4096, 4097, 8300]),
    # with enough groups the items keep 4096 rows
    ("bf16-d128-G4-split4096", dict(n_layers=2, batch=4, n_q_heads=32, n_kv_heads=8,
                                    head_dim=128, dtype="bf16", seed=53), [4097, 8300]),
    ("bf16-d128-G1", dict(n_layers=2, batch=2, n_q_heads=2, n_kv_heads=2, head_dim=128,
                          dtype="bf16", seed=48), [0, 129]),
    ("bf16-d128-G2", dict(n_layers=2, batch=1, n_q_heads=4, n_kv_heads=2, head_dim=128,
                          dtype="bf16", kv_dist="scaled_sinks", seed=49), [31, 4095]),
]


@pytest.mark.parametrize("name,over,lens0", DECODE_SHAPES, ids=[c[0] for c in DECODE_SHAPES])
def test_decode_matches_oracle_over_steps(lib, name, over, lens0):
    wl = synth.WORKLOADS["tiny"].replace(**over)
    steps = 3
    caps = [n + steps + 2 for n in lens0]
    kc, vc = zip(*[synth.decode_caches(wl, i, caps[i]) for i in range(wl.n_layers)])
    s = Session(lib, wl, range(wl.n_layers), caps, lens0, kc, vc)
    rows_k = [[[synth.to_f64(kc[i][b, h, :lens0[i]]) for h in range(wl.n_kv_heads)]
               for b in range(wl.batch)] for i in range(wl.n_layers)]
    rows_v = [[[synth.to_f64(vc[i][b, h, :lens0[i]]) for h in range(wl.n_kv_heads)]
               for b in range(wl.batch)] for i in range(wl.n_layers)]
    for t in range(steps):
        q, kn, vn = synth.decode_inputs(wl, t)
        got = s.step(q, kn, vn)
        ref = _oracle_step(wl, rows_k, rows_v, q, kn, vn)
        C.assert_decode_close(got, ref)
        assert int(s.status.item()) == 0
        assert s.lens.cpu().tolist() == [n + t + 1 for n in lens0]
        for i in range(wl.n_layers):
            # the appended rows are the new token's rows, bit for bit
            assert torch.equal(s.k[i][:, :, lens0[i] + t].cpu(), kn[i])
            assert torch.equal(s.v[i][:, :, lens0[i] + t].cpu(), vn[i])


def test_decode_single_row_is_value(lib):
    # an empty cache: the new token attends only to itself, o = v_new (Sec. 4.1)
    wl = synth.WORKLOADS["tiny"].replace(n_layers=1, dtype="bf16", head_dim=128, seed=44)
    kc, vc = synth.decode_caches(wl, 0, 4)
    s = Session(lib, wl, [0], [4], [0], [kc], [vc])
    q, kn, vn = synth.decode_inputs(wl, 0)
    got = s.step(q, kn, vn)
    G = wl.group
    for h in range(wl.n_kv_heads):
        for g in range(G):
            np.testing.assert_array_equal(got[0, 0, h * G + g], vn[0, 0, h].float().numpy())


def test_decode_full_cache_reports_and_skips(lib):
    wl = synth.WORKLOADS["tiny"].replace(n_layers=2, seed=45)
    caps = [10, 10]
    kc, vc = zip(*[synth.decode_caches(wl, i, 10) for i in range(2)])
    s = Session(lib, wl, range(2), caps, [10, 4], kc, vc)
    q, kn, vn = synth.decode_inputs(wl, 0)
    got = s.step(q, kn, vn)
    assert int(s.status.item()) == lib.EFULL
    assert s.lens.cpu().tolist() == [10, 5]
    assert np.all(got[0] == 0.0) and np.any(got[1] != 0.0)
    assert torch.equal(s.k[0].cpu(), kc[0])


def test_decode_full_cache_bf16_d128(lib):
    # bf16, d = 128: a full layer is skipped and reported
    wl = synth.WORKLOADS["tiny"].replace(n_layers=2, dtype="bf16", head_dim=128, n_q_heads=8,
                                         n_kv_heads=2, seed=50)
    caps = [300, 300]
    kc, vc = zip(*[synth.decode_caches(wl, i, 300) for i in range(2)])
    s = Session(lib, wl, range(2), caps, [300, 200], kc, vc)
    q, kn, vn = synth.decode_inputs(wl, 0)
    got = s.step(q, kn, vn)
    assert int(s.status.item()) == lib.EFULL
    assert s.lens.cpu().tolist() == [300, 201]
    assert np.all(got[0] == 0.0)
    rows_k = [[[synth.to_f64(kc[1][b, h, :200]) for h in range(wl.n_kv_heads)]
               for b in range(wl.batch)]]
    rows_v = [[[synth.to_f64(vc[1][b, h, :200]) for h in range(wl.n_kv_heads)]
               for b in range(wl.batch)]]
    ref = _oracle_step(wl, rows_k, rows_v, q[1:], kn[1:], vn[1:])
    C.assert_decode_close(got[1:], ref)
    assert torch.equal(s.k[0].cpu(), kc[0])


def _compress_all(lib, wl, budgets, cap_extra, device_gen="cpu"):
    outs, inputs = [], []
    for layer in range(wl.n_layers):
        q_win, k, v = (t.to(DEV) for t in C.layer_inputs(wl, layer, device_gen))
        outs.append(C.run_compress(lib, wl, budgets[layer], q_win, k, v, cap_extra=cap_extra,
                                   scores=False))
        inputs.append((q_win, k, v))
    return outs, inputs


def test_end_to_end_tiny_against_oracle(lib):
    # compress all layers with RippleKV budgets, then decode; the oracle runs
    # its own compression (its own scores and selection) and its own decode
    wl = synth.WORKLOADS["tiny"]
    s_prof = synth.sensitivity_profile(wl)
    budgets = lib.ripple_alloc_budgets(s_prof, wl.ratio, wl.gamma, wl.global_budget)
    outs, inputs = _compress_all(lib, wl, budgets, cap_extra=2)
    caps = [o["k_out"].shape[2] for o in outs]
    sess = Session(lib, wl, range(wl.n_layers), caps, [o["n"] for o in outs],
                   [o["k_out"] for o in outs], [o["v_out"] for o in outs])
    scale = 1.0 / np.sqrt(wl.head_dim)
    rows_k, rows_v = [], []
    for layer, (q_win, k, v) in enumerate(inputs):
        rk, rv = [], []
        for b in range(wl.batch):
            ck, cv = [], []
            for h in range(wl.n_kv_heads):
                qf, kf, vf = C.unit_f64(wl, q_win, k, v, b, h)
                ref = O.compress_unit(qf, kf, vf, budgets[layer], wl.window, scale,
                                      wl.pool_kernel)
                ck.append(ref["k_out"])
                cv.append(ref["v_out"])
            rk.append(ck)
            rv.append(cv)
        rows_k.append(rk)
        rows_v.append(rv)
    for t in range(wl.decode_steps + 1):
        q, kn, vn = synth.decode_inputs(wl, t)
        got = sess.step(q, kn, vn)
        ref = _oracle_step(wl, rows_k, rows_v, q, kn, vn)
        C.assert_decode_close(got, ref)


def test_budget_at_least_T_reproduces_full_attention_exactly(lib):
    # b_l >= T keeps every token: the compressed cache equals the full cache and
    # decoding over it equals decoding over the uncompressed cache bit for bit
    wl = synth.WORKLOADS["tiny"].replace(dtype="bf16", head_dim=128, n_layers=2, seed=46)
    budgets = [wl.seq_len, 10 * wl.seq_len]
    outs, inputs = _compress_all(lib, wl, budgets, cap_extra=1)
    full_k, full_v = [], []
    for (q_win, k, v), o in zip(inputs, outs):
        assert torch.equal(o["k_out"][:, :, :wl.seq_len], k)
        assert torch.equal(o["v_out"][:, :, :wl.seq_len], v)
        fk = torch.zeros_like(o["k_out"])
        fv = torch.zeros_like(o["v_out"])
        fk[:, :, :wl.seq_len] = k
        fv[:, :, :wl.seq_len] = v
        full_k.append(fk)
        full_v.append(fv)
    caps = [wl.seq_len + 1] * 2
    a = Session(lib, wl, range(2), caps, [wl.seq_len] * 2, [o["k_out"] for o in outs],
                [o["v_out"] for o in outs])
    b = Session(lib, wl, range(2), caps, [wl.seq_len] * 2, full_k, full_v)
    q, kn, vn = synth.decode_inputs(wl, 0)
    got_a = a.step(q, kn, vn)
    got_b = b.step(q, kn, vn)
    np.testing.assert_array_equal(got_a, got_b)
    rows_k = [[[synth.to_f64(inp[1][bb, h]) for h in range(wl.n_kv_heads)]
               for bb in range(wl.batch)] for inp in inputs]
    rows_v = [[[synth.to_f64(inp[2][bb, h]) for h in range(wl.n_kv_heads)]
               for bb in range(wl.batch)] for inp in inputs]
    ref = _oracle_step(wl, rows_k, rows_v, q, kn, vn)
    C.assert_decode_close(got_a, ref)


def _sample_groups(wl, lens0):
    """A fixed sample of (layer, b, kv head) groups: the first and last, the
    longest cache, and one in the middle."""
    L, B, H = wl.n_layers, wl.batch, wl.n_kv_heads
    return sorted({(0, 0, 0), (int(np.argmax(lens0)), B - 1, H - 1), (L - 1, B // 2, H // 2),
                   (L // 2, (B - 1) // 3, (H - 1) // 3)})


@pytest.mark.parametrize("name", ["llama8b-32k", "mistral7b-16k", "llama70b-128k"])
def test_full_size_decode_sampled(lib, name):
    # every layer's ragged cache at its RippleKV size, two decode steps over all
    # layers in one call (the benchmark's launch); the oracle checks a sample of
    # (layer, batch, kv head) groups
    wl = synth.WORKLOADS[name]
    s_prof = synth.sensitivity_profile(wl)
    budgets = lib.ripple_alloc_budgets(s_prof, wl.ratio, wl.gamma, wl.global_budget)
    lens0 = [lib.ripple_keep_count(b, wl.seq_len, wl.window) for b in budgets]
    caps = [n + 4 for n in lens0]
    kc, vc = zip(*[synth.decode_caches(wl, i, caps[i], DEV) for i in range(wl.n_layers)])
    s = Session(lib, wl, range(wl.n_layers), caps, lens0, kc, vc)
    sample = _sample_groups(wl, lens0)
    G = wl.group
    scale = 1.0 / np.sqrt(wl.head_dim)
    hist = {key: (synth.to_f64(kc[key[0]][key[1], key[2], :lens0[key[0]]]),
                  synth.to_f64(vc[key[0]][key[1], key[2], :lens0[key[0]]])) for key in sample}
    for t in range(2):
        q, kn, vn = synth.decode_inputs(wl, t, DEV)
        got = s.step(q, kn, vn)
        assert int(s.status.item()) == 0
        for (l, b, h) in sample:
            rk, rv = hist[(l, b, h)]
            rk = np.vstack([rk, synth.to_f64(kn[l, b, h])[None]])
            rv = np.vstack([rv, synth.to_f64(vn[l, b, h])[None]])
            hist[(l, b, h)] = (rk, rv)
            ref = O.decode_attention(synth.to_f64(q[l, b, h * G:(h + 1) * G]), rk, rv, scale)
            C.assert_decode_close(got[l, b, h * G:(h + 1) * G], ref)
    assert s.lens.cpu().tolist() == [n + 2 for n in lens0]
    del s, kc, vc
    torch.cuda.empty_cache()


def _garbage_(t, seed):
    g = torch.Generator(device=t.device)
    g.manual_seed(seed)
    t.copy_(torch.randint(0, 256, t.shape, generator=g, device=t.device, dtype=torch.uint8))


def test_workspace_contents_do_not_matter(lib):
    # The workspace is filled with random bytes before every step (as memory
    # freed by one tensor and handed to the next by an allocator would be);
    # each call zeroes the counters it uses, so results match the oracle.
    wl = synth.WORKLOADS["tiny"].replace(n_layers=3, batch=2, n_q_heads=8, n_kv_heads=2,
                                         head_dim=128, dtype="bf16", kv_dist="scaled_sinks",
                                         seed=51)
    lens0 = [300, 4097, 9000]  # single-item and split groups (group counters in use)
    caps = [n + 4 for n in lens0]
    kc, vc = zip(*[synth.decode_caches(wl, i, caps[i]) for i in range(wl.n_layers)])
    s = Session(lib, wl, range(wl.n_layers), caps, lens0, kc, vc)
    rows_k = [[[synth.to_f64(kc[i][b, h, :lens0[i]]) for h in range(wl.n_kv_heads)]
               for b in range(wl.batch)] for i in range(wl.n_layers)]
    rows_v = [[[synth.to_f64(vc[i][b, h, :lens0[i]]) for h in range(wl.n_kv_heads)]
               for b in range(wl.batch)] for i in range(wl.n_layers)]
    for t in range(3):
        _garbage_(s.ws, 100 + t)
        q, kn, vn = synth.decode_inputs(wl, t)
        got = s.step(q, kn, vn)
        assert int(s.status.item()) == 0
        C.assert_decode_close(got, _oracle_step(wl, rows_k, rows_v, q, kn, vn))
    assert s.lens.cpu().tolist() == [n + 3 for n in lens0]


def test_workspace_reallocated_at_the_same_address(lib):
    # Free the workspace, let another tensor take its memory and write into
    # it, free that and allocate a new workspace (the caching allocator hands
    # out the same block): decode still equals a run on a fresh workspace.
    wl = synth.WORKLOADS["tiny"].replace(n_layers=2, batch=1, n_q_heads=8, n_kv_heads=2,
                                         head_dim=128, dtype="bf16", seed=52)
    lens0 = [5000, 130]
    caps = [n + 4 for n in lens0]
    kc, vc = zip(*[synth.decode_caches(wl, i, caps[i]) for i in range(wl.n_layers)])
    a = Session(lib, wl, range(2), caps, lens0, kc, vc)
    b = Session(lib, wl, range(2), caps, lens0, kc, vc)
    nbytes = a.ws.numel()
    reused = 0
    for t in range(3):
        q, kn, vn = synth.decode_inputs(wl, t)
        want = a.step(q, kn, vn)
        addr = b.ws.data_ptr()
        b.ws = None
        other = torch.empty(nbytes, dtype=torch.uint8, device=DEV)
        _garbage_(other, 200 + t)
        del other
        b.ws = torch.empty(nbytes, dtype=torch.uint8, device=DEV)
        reused += b.ws.data_ptr() == addr
        got = b.step(q, kn, vn)
        assert int(b.status.item()) == 0
        np.testing.assert_array_equal(got, want)
    print(f"workspace handed back at the same address in {reused} of 3 steps")
