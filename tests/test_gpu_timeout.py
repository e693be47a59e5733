"""The bounded in-kernel waits give up, report RIPPLE_ETIMEOUT and leave the
GPU usable. ripple_set_wait_limit_cycles makes every wait of the next launches
give up after a few cycles (no fault, no hang: each wait still ends, and a
block that gave up waits for its own bulk copies before it leaves, and frees
its tensor memory); the call must come back within seconds with
RIPPLE_ETIMEOUT in the device status, and the next call at the default limit
must match the oracle again.

A wait gives up only after a poll of its mbarrier has come back empty; one
poll may suspend the thread until the phase completes or a hardware time
limit passes, so waits on a bulk copy that lands within that limit never give
up. The calls tested here also wait on flags other thread blocks raise (the
decode's counter initialisation, the scoring's row statistics), which do."""
import time

import numpy as np
import pytest
import torch

from oracle import ripple_oracle as O
from paper_2608_08684_gb300 import synth
from tests import gpu_common as C

pytestmark = pytest.mark.gpu
DEV = "cuda"
TINY_LIMIT = 100  # SM cycles: far below one DRAM round trip


class _ShortWaits:
    def __init__(self, lib):
        self.lib = lib

    def __enter__(self):
        self.prev = self.lib.ripple_set_wait_limit_cycles(TINY_LIMIT)
        return self

    def __exit__(self, *exc):
        self.lib.ripple_set_wait_limit_cycles(0)


def _timed_sync():
    t = time.perf_counter()
    torch.cuda.synchronize()
    return time.perf_counter() - t


def test_wait_limit_setter_round_trips(lib):
    prev = lib.ripple_set_wait_limit_cycles(12345)
    try:
        assert lib.ripple_set_wait_limit_cycles(0) == 12345
        assert lib.ripple_set_wait_limit_cycles(0) == 4_000_000_000
    finally:
        lib.ripple_set_wait_limit_cycles(0)
    assert prev == 4_000_000_000


def test_compress_layers_times_out_then_recovers(lib):
    # two layers of the 32k workload's shape: the tensor-core scoring (waits
    # on its TMA ring, TMEM accumulators and other blocks' row statistics) and
    # the gather (waits on its bulk copies)
    wl = synth.WORKLOADS["llama8b-32k"].replace(n_layers=2)
    L, B, H, d = wl.n_layers, wl.batch, wl.n_kv_heads, wl.head_dim
    budgets = [1500, 700]
    desc = lib.layer_desc(B, wl.n_q_heads, H, d, wl.seq_len, wl.window, wl.pool_kernel, "max",
                          wl.torch_dtype)
    ins = [C.layer_inputs(wl, l, DEV) for l in range(L)]
    ns = [lib.ripple_keep_count(b, wl.seq_len, wl.window) for b in budgets]

    def run():
        k_out = [torch.zeros(B, H, n, d, dtype=wl.torch_dtype, device=DEV) for n in ns]
        v_out = [torch.zeros_like(x) for x in k_out]
        idx = [torch.full((B * H * n,), -1, dtype=torch.int32, device=DEV) for n in ns]
        tables = lib.CompressTables([x[0] for x in ins], [x[1] for x in ins],
                                    [x[2] for x in ins], k_out, v_out, idx)
        ws = torch.empty(lib.ripple_compress_layers_workspace_bytes(desc, L), dtype=torch.uint8,
                         device=DEV)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        lib.ripple_compress_layers(desc, budgets, tables, ws, dev_status=status)
        return status, k_out, v_out, idx

    torch.cuda.synchronize()
    with _ShortWaits(lib):
        status, *_ = run()
    assert _timed_sync() < 10.0
    assert int(status.item()) == lib.ETIMEOUT
    # default limit, fresh workspace and outputs: parity with the oracle
    status, k_out, v_out, idx = run()
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    agree = total = 0
    for l in range(L):
        q, k, v = ins[l]
        out = {"n": ns[l], "idx": idx[l].view(B, H, ns[l]), "k_out": k_out[l],
               "v_out": v_out[l], "scores": None}
        for b, h in [(0, 0), (B - 1, H - 1)]:
            a, t = C.check_compress_unit(wl, out, q, k, v, b, h, budgets[l])
            agree += a
            total += t
    assert agree >= 0.999 * total


def test_decode_times_out_then_recovers(lib):
    wl = synth.WORKLOADS["tiny"].replace(n_layers=2, batch=2, n_q_heads=8, n_kv_heads=2,
                                         head_dim=128, dtype="bf16", kv_dist="scaled_sinks",
                                         seed=61)
    # long caches: many sub-chunk stages per work item, so that stage waits
    # depend on the other role's progress
    lens0 = [24000, 9000]
    caps = [n + 2 for n in lens0]
    desc = lib.decode_desc(2, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.torch_dtype)
    ws = torch.empty(lib.ripple_decode_workspace_bytes(desc, caps), dtype=torch.uint8,
                     device=DEV)
    q, kn, vn = (t.to(DEV) for t in synth.decode_inputs(wl, 0))

    def run():
        kc, vc = zip(*[synth.decode_caches(wl, i, caps[i], DEV) for i in range(2)])
        tables = lib.DecodeTables(list(kc), list(vc))
        lens = torch.tensor(lens0, dtype=torch.int32, device=DEV)
        out = torch.empty(2, wl.batch, wl.n_q_heads, wl.head_dim, device=DEV)
        status = torch.zeros(1, dtype=torch.int32, device=DEV)
        lib.ripple_decode_attn(desc, q, kn, vn, tables, lens, out, ws, dev_status=status)
        return status, out, kc, vc

    torch.cuda.synchronize()
    # Whether a wait outlasts the bound depends on timing (an mbarrier wait is
    # suspended in hardware and may return only when its phase completes), so
    # the short-bound call is repeated until one of its waits gives up.
    seen = []
    for _ in range(5):
        with _ShortWaits(lib):
            status, *_ = run()
        assert _timed_sync() < 10.0
        seen.append(int(status.item()))
        if seen[-1] == lib.ETIMEOUT:
            break
    assert seen[-1] == lib.ETIMEOUT and set(seen) <= {0, lib.ETIMEOUT}, seen
    # the same workspace (left as the timed-out call left it), default limit
    status, out, kc, vc = run()
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    got = out.cpu().numpy()
    G, scale = wl.group, 1.0 / np.sqrt(wl.head_dim)
    for l in range(2):
        for b in range(wl.batch):
            for h in range(wl.n_kv_heads):
                rk = np.vstack([synth.to_f64(kc[l][b, h, :lens0[l]]), synth.to_f64(kn[l, b, h])[None]])
                rv = np.vstack([synth.to_f64(vc[l][b, h, :lens0[l]]), synth.to_f64(vn[l, b, h])[None]])
                ref = O.decode_attention(synth.to_f64(q[l, b, h * G:(h + 1) * G]), rk, rv, scale)
                C.assert_decode_close(got[l, b, h * G:(h + 1) * G], ref)
