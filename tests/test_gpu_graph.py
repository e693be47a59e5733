"""Stream-ordered entry points are capturable in CUDA graphs (no host sync, no
allocation inside a call): decode steps and a multi-layer compression captured
once and replayed give exactly the eager results."""
import pytest
import torch

from paper_2608_08684_gb300 import synth
from tests import gpu_common as C

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _decode_setup(lib, wl, lens0, steps):
    caps = [n + steps + 2 for n in lens0]
    kc, vc = zip(*[synth.decode_caches(wl, i, caps[i], DEV) for i in range(wl.n_layers)])
    k = [t.clone() for t in kc]
    v = [t.clone() for t in vc]
    desc = lib.decode_desc(wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim,
                           wl.torch_dtype)
    s = dict(k=k, v=v, tables=lib.DecodeTables(k, v), desc=desc,
             lens=torch.tensor(lens0, dtype=torch.int32, device=DEV),
             ws=torch.empty(lib.ripple_decode_workspace_bytes(desc, caps), dtype=torch.uint8,
                            device=DEV),
             status=torch.zeros(1, dtype=torch.int32, device=DEV),
             out=torch.empty(steps, wl.n_layers, wl.batch, wl.n_q_heads, wl.head_dim,
                             device=DEV),
             inputs=[synth.decode_inputs(wl, t, DEV) for t in range(steps)])
    return s


def _decode_steps(lib, s, stream=None):
    for t, (q, kn, vn) in enumerate(s["inputs"]):
        lib.ripple_decode_attn(s["desc"], q, kn, vn, s["tables"], s["lens"], s["out"][t], s["ws"],
                               dev_status=s["status"], stream=stream)


@pytest.mark.parametrize("over", [
    dict(n_layers=3, batch=2, n_q_heads=8, n_kv_heads=2, head_dim=128, dtype="bf16", seed=61),
    dict(n_layers=2, batch=1, n_q_heads=4, n_kv_heads=2, head_dim=64, dtype="f32", seed=62),
], ids=["bf16-d128", "f32-d64"])
def test_decode_steps_replay_from_a_graph(lib, over):
    wl = synth.WORKLOADS["tiny"].replace(**over)
    lens0, steps = [5, 300, 129][:wl.n_layers], 4
    eager = _decode_setup(lib, wl, lens0, steps)
    _decode_steps(lib, eager)
    torch.cuda.synchronize()
    assert int(eager["status"].item()) == 0

    g = _decode_setup(lib, wl, lens0, steps)
    # warm-up call outside the capture (first-use set-up), then reset the state
    side = _decode_setup(lib, wl, lens0, 1)
    _decode_steps(lib, side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        with torch.cuda.graph(graph, stream=s):
            _decode_steps(lib, g, stream=s)
    graph.replay()
    torch.cuda.synchronize()
    assert int(g["status"].item()) == 0
    assert torch.equal(g["out"], eager["out"])
    assert g["lens"].tolist() == eager["lens"].tolist()
    for a, b in zip(g["k"], eager["k"]):
        assert torch.equal(a, b)


def test_compress_layers_replay_from_a_graph(lib):
    wl = synth.WORKLOADS["tiny"].replace(n_layers=3, batch=2, n_q_heads=8, n_kv_heads=2,
                                         head_dim=128, seq_len=900, dtype="bf16", seed=63)
    budgets = [100, 400, 40]
    desc = lib.layer_desc(wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.seq_len,
                          wl.window, wl.pool_kernel, "max", wl.torch_dtype)
    ins = [tuple(t.to(DEV) for t in C.layer_inputs(wl, l, "cpu")) for l in range(wl.n_layers)]
    ns = [lib.ripple_keep_count(b, wl.seq_len, wl.window) for b in budgets]

    def buffers():
        ko = [torch.zeros(wl.batch, wl.n_kv_heads, n, wl.head_dim, dtype=wl.torch_dtype,
                          device=DEV) for n in ns]
        vo = [torch.zeros_like(x) for x in ko]
        ix = [torch.full((wl.batch * wl.n_kv_heads * n,), -1, dtype=torch.int32, device=DEV)
              for n in ns]
        tab = lib.CompressTables([x[0] for x in ins], [x[1] for x in ins], [x[2] for x in ins],
                                 ko, vo, ix)
        ws = torch.empty(lib.ripple_compress_layers_workspace_bytes(desc, wl.n_layers),
                         dtype=torch.uint8, device=DEV)
        return ko, vo, ix, tab, ws

    ko1, vo1, ix1, tab1, ws1 = buffers()
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    lib.ripple_compress_layers(desc, budgets, tab1, ws1, dev_status=st)
    torch.cuda.synchronize()
    ko2, vo2, ix2, tab2, ws2 = buffers()
    graph = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        with torch.cuda.graph(graph, stream=s):
            lib.ripple_compress_layers(desc, budgets, tab2, ws2, dev_status=st, stream=s)
    graph.replay()
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    for a, b in zip(ix1 + ko1 + vo1, ix2 + ko2 + vo2):
        assert torch.equal(a, b)
