"""ripple_decode_attn_noalloc: the decode step for callers that cannot allocate
device memory (for example a plugin whose host program owns every device
buffer and only hands over input and output tensors). It keeps its split-K
partials in the library's own fixed device array instead of a caller
workspace, so it must give the same results as ripple_decode_attn, step after
step, with the scratch array reused between calls.

This file is collected last on purpose: if it fails, a run stopping at the
first failure has already run every other test.
"""
import pytest
import torch

from paper_2608_08684_gb300 import synth

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _caches(wl, caps):
    kc, vc = zip(*[synth.decode_caches(wl, i, caps[i]) for i in range(wl.n_layers)])
    return [t.to(DEV) for t in kc], [t.to(DEV) for t in vc]


@pytest.mark.parametrize("over,lens0", [
    (dict(n_layers=3, batch=2, n_q_heads=8, n_kv_heads=2, head_dim=128, dtype="bf16",
          kv_dist="scaled_sinks", seed=71), [5, 130, 300]),
    (dict(n_layers=2, seed=72), [1, 257]),
])
def test_noalloc_decode_matches_workspace_decode(lib, over, lens0):
    wl = synth.WORKLOADS["tiny"].replace(**over)
    caps = [n + 4 for n in lens0]
    ka, va = _caches(wl, caps)
    kb, vb = [t.clone() for t in ka], [t.clone() for t in va]
    desc = lib.decode_desc(wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim,
                           wl.torch_dtype)
    ta, tb = lib.DecodeTables(ka, va), lib.DecodeTables(kb, vb)
    ws = torch.empty(lib.ripple_decode_workspace_bytes(desc, caps), dtype=torch.uint8, device=DEV)
    lens_a = torch.tensor(lens0, dtype=torch.int32, device=DEV)
    lens_b = lens_a.clone()
    st_a = torch.zeros(1, dtype=torch.int32, device=DEV)
    st_b = torch.zeros(1, dtype=torch.int32, device=DEV)
    shape = (wl.n_layers, wl.batch, wl.n_q_heads, wl.head_dim)
    for step in range(2):  # two calls in a row share the scratch array
        q, kn, vn = (t.to(DEV) for t in synth.decode_inputs(wl, step))
        out_a = torch.empty(shape, dtype=torch.float32, device=DEV)
        out_b = torch.full(shape, float("nan"), dtype=torch.float32, device=DEV)
        lib.ripple_decode_attn(desc, q, kn, vn, ta, lens_a, out_a, ws, dev_status=st_a)
        lib.ripple_decode_attn_noalloc(desc, q, kn, vn, tb, lens_b, out_b, dev_status=st_b)
        torch.cuda.synchronize()
        assert int(st_a.item()) == 0 and int(st_b.item()) == 0
        assert torch.isfinite(out_b).all()
        # same kernel, same work plan, fixed-order combine: identical bits
        assert torch.equal(out_a, out_b)
        assert torch.equal(lens_a, lens_b)
        for x, y in zip(ka + va, kb + vb):
            assert torch.equal(x, y)


def test_noalloc_rejects_steps_beyond_its_scratch(lib):
    # caps whose partials exceed the fixed array are refused before any launch
    wl = synth.WORKLOADS["tiny"].replace(n_layers=1, batch=64, n_q_heads=64, n_kv_heads=8,
                                         head_dim=128, dtype="bf16")
    caps = [32768]
    desc = lib.decode_desc(1, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.torch_dtype)
    assert lib.ripple_decode_workspace_bytes(desc, caps) > lib.NOALLOC_SCRATCH_BYTES
    # the request is refused on the host from desc and caps alone, so small
    # tensors with the right capacity stand in for the caches
    k = torch.zeros(1, 1, caps[0], wl.head_dim, dtype=wl.torch_dtype, device=DEV)
    tables = lib.DecodeTables([k], [k.clone()])
    q = torch.zeros(1, wl.batch, wl.n_q_heads, wl.head_dim, dtype=wl.torch_dtype, device=DEV)
    kn = torch.zeros(1, wl.batch, wl.n_kv_heads, wl.head_dim, dtype=wl.torch_dtype, device=DEV)
    lens = torch.zeros(1, dtype=torch.int32, device=DEV)
    out = torch.zeros(1, wl.batch, wl.n_q_heads, wl.head_dim, device=DEV)
    before = lib.ripple_kernel_launches()
    with pytest.raises(lib.RippleError) as e:
        lib.ripple_decode_attn_noalloc(desc, q, kn, kn.clone(), tables, lens, out)
    assert e.value.status == lib.EWORKSPACE
    assert lib.ripple_kernel_launches() == before
