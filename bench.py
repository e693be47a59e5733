#!/usr/bin/env python3
"""Benchmark of the RippleKV serving hot path on GB300.

One step = the whole path on one synthetic batch: host budget allocation
(Eqs. 9-12), compression of every layer (scoring, pooling, top-k, gather) and
the workload's decode steps over the ragged caches, all through the C ABI.

Default workload: the Llama-3-8B-shaped 32k stack (32 layers, 32 q / 8 KV
heads, d = 128, batch 4, T = 32768, bf16, average budget 1024, ratio 8, 128
decode steps). Inputs are synthetic (seeded), generated on the device and
resident in HBM when the timed region starts; per layer K + V is 537 MB, far
above the 129 MB L2, so no flush is needed between steps.

Output: one JSON line (rank 0). `value` = prompt tokens compressed and then
decoded per second over whole steps (B * T * ranks / step time). Extra keys
break the step down: compression-only tokens/s and decode-attention GB/s, each
against the measured HBM copy bandwidth.

--impl reference times the CPU oracle (the test-infrastructure restatement of
the paper) on a bounded sample of the same workload, extrapolated to a step.

--case compress|decode times one entry point of the serving path alone;
--case perturb|kl times the offline profiling kernels (Sec. 4.3: Eq. 6 on one
layer's V cache, Eq. 7 for one perturbed run per layer); each prints one JSON
line with its algorithmic bytes and fraction of the measured HBM bandwidth.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

HBM_FALLBACK_GBS = 6800.0
REASON_BITS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
               0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
               0x100: "display_clock_setting"}
# the benchmark's metric (both arms print it)
METRIC = "compressed-prefill tokens/s; ragged decode-attn HBM GB/s vs GB300 peak"


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="llama8b-32k")
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the other workloads and the serving-loop measurement")
    ap.add_argument("--cpu-seconds", type=float, default=15.0,
                    help="target CPU seconds of the oracle sample")
    ap.add_argument("--case", choices=["compress", "attn", "decode", "perturb", "kl", "serve"],
                    default=None,
                    help="time one entry point alone (one layer / one decode step / the "
                         "profiling kernels: Eq. 6 perturbation of one layer's V cache, Eq. 7 "
                         "window KL of every layer's perturbed run; serve: the per-layer "
                         "decode loop with stand-in projections in a CUDA graph), e.g. as a "
                         "small ncu target; prints one JSON line")
    ap.add_argument("--vocab", type=int, default=128256,
                    help="--case kl: vocabulary size (128256: Llama-3)")
    ap.add_argument("--repeat", type=int, default=10, help="calls timed in --case mode")
    ap.add_argument("--layers", type=int, default=1,
                    help="--case compress: compress this many layers in one "
                         "ripple_compress_layers call (budgets of the largest-budget layers, "
                         "all reading that layer's K/V so the device footprint stays one layer's)")
    return ap.parse_args()


def run_case(args):
    """Single-entry-point timing: compression of the workload's largest-budget
    layer, or one decode step over every layer's ragged cache (seeded caches
    at the RippleKV sizes). Inputs stay within a few GB of device memory."""
    import torch

    from paper_2608_08684_gb300 import build as _build
    from paper_2608_08684_gb300 import synth
    _build.build_library()
    from paper_2608_08684_gb300 import ripple as R
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    wl = synth.WORKLOADS[args.workload]
    L, B, Hq, Hkv, d, e = (wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim,
                           wl.elem_bytes)
    budgets = R.ripple_alloc_budgets(synth.sensitivity_profile(wl), wl.ratio, wl.gamma,
                                     wl.global_budget)
    n_keep = [R.ripple_keep_count(b, wl.seq_len, wl.window) for b in budgets]
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    times = []
    if args.case in ("perturb", "kl"):
        return run_profile_case(args, R, synth, wl, dev)
    if args.case == "attn":
        return run_attn_case(args, R, synth, wl, dev, budgets, n_keep)
    if args.case == "serve":
        line = {"case": "serve", "workload": wl.name}
        line.update(serving_loop_measure(R, synth, wl, dev, min(args.repeat * 4, wl.decode_steps)))
        print(json.dumps(line), flush=True)
        return
    if args.case == "compress":
        layer = max(range(L), key=lambda i: budgets[i])
        q_win = synth.layer_window_queries(wl, layer, dev)
        k = synth.layer_keys(wl, layer, dev)
        v = synth.layer_values(wl, layer, dev)
        desc = R.layer_desc(B, Hq, Hkv, d, wl.seq_len, wl.window, wl.pool_kernel, "max",
                            wl.torch_dtype)
        n = n_keep[layer]
        ws = torch.empty(R.ripple_compress_workspace_bytes(desc), dtype=torch.uint8, device=dev)
        k_out = torch.empty(B, Hkv, n, d, dtype=wl.torch_dtype, device=dev)
        v_out = torch.empty_like(k_out)
        idx = torch.empty(B * Hkv * n, dtype=torch.int32, device=dev)
        nbytes = B * Hkv * d * e * (wl.seq_len + 3 * n) + B * Hq * wl.window * d * e
        if args.layers > 1:
            # several layers in one call: the args.layers largest-budget
            # layers, each with its own inputs
            lay = sorted(range(L), key=lambda i: -budgets[i])[:args.layers]
            outs = [(torch.empty(B, Hkv, n_keep[i], d, dtype=wl.torch_dtype, device=dev),
                     torch.empty(B, Hkv, n_keep[i], d, dtype=wl.torch_dtype, device=dev),
                     torch.empty(B * Hkv * n_keep[i], dtype=torch.int32, device=dev))
                    for i in lay]
            ins = [(synth.layer_window_queries(wl, i, dev), synth.layer_keys(wl, i, dev),
                    synth.layer_values(wl, i, dev)) for i in lay]
            tabs = R.CompressTables([x[0] for x in ins], [x[1] for x in ins], [x[2] for x in ins],
                                    [o[0] for o in outs], [o[1] for o in outs],
                                    [o[2] for o in outs])
            ws = torch.empty(R.ripple_compress_layers_workspace_bytes(desc, len(lay)),
                             dtype=torch.uint8, device=dev)
            nbytes = sum(B * Hkv * d * e * (wl.seq_len + 3 * n_keep[i]) + B * Hq * wl.window * d * e
                         for i in lay)
        for i in range(args.repeat + 2):
            a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            if args.layers > 1:
                R.ripple_compress_layers(desc, [budgets[i] for i in lay], tabs, ws,
                                         dev_status=status)
            else:
                R.ripple_compress_layer(desc, budgets[layer], q_win, k, v, k_out, v_out, idx, ws,
                                        dev_status=status)
            b_.record()
            if i >= 2:
                times.append((a, b_))
        what = (f"compress {len(lay)} layers in one call (layers {lay}, each with its own "
                f"inputs)" if args.layers > 1 else
                f"compress layer {layer} (budget {budgets[layer]}, n {n})")
    else:
        steps = args.repeat
        caps = [n + steps + 1 for n in n_keep]
        kc, vc = zip(*[synth.decode_caches(wl, i, caps[i], dev) for i in range(L)])
        tables = R.DecodeTables(list(kc), list(vc))
        ddesc = R.decode_desc(L, B, Hq, Hkv, d, wl.torch_dtype)
        dws = torch.empty(R.ripple_decode_workspace_bytes(ddesc, caps), dtype=torch.uint8,
                          device=dev)
        lens0 = torch.tensor(n_keep, dtype=torch.int32, device=dev)
        lens = lens0.clone()
        q, kn, vn = synth.decode_inputs(wl, 0, dev)
        out = torch.empty(L, B, Hq, d, device=dev)
        # `steps` decode steps back to back (lengths n .. n + steps - 1), timed
        # as one block after two untimed warm-up steps
        nbytes = sum(sum(B * Hkv * 2 * (n + s + 1) * d * e for n in n_keep)
                     + L * B * Hq * d * (e + 4) + L * B * Hkv * d * e * 4
                     for s in range(steps)) // steps
        for _ in range(2):
            R.ripple_decode_attn(ddesc, q, kn, vn, tables, lens, out, dws, dev_status=status)
        lens.copy_(lens0)
        torch.cuda.synchronize()
        a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(steps):
            R.ripple_decode_attn(ddesc, q, kn, vn, tables, lens, out, dws, dev_status=status)
        b_.record()
        times.append((a, b_))
        what = (f"{steps} decode steps back to back over {L} layers, lens from "
                f"{min(n_keep)}..{max(n_keep)}")
    torch.cuda.synchronize()
    assert int(status.item()) == 0, int(status.item())
    ms = statistics.mean(a.elapsed_time(b) for a, b in times)
    if args.case == "decode":
        ms /= args.repeat  # one block of back-to-back steps
    hbm, src = measured_peaks()
    gbs = nbytes / (ms / 1e3) / 1e9
    print(json.dumps({"case": args.case, "workload": wl.name, "what": what, "calls": args.repeat if args.case == "decode" else len(times),
                      "ms_per_call": round(ms, 5), "bytes_per_call": nbytes,
                      "gbs": round(gbs, 1), "frac_hbm": round(gbs / hbm, 4),
                      "peak_source": src}), flush=True)


def run_attn_case(args, R, synth, wl, dev, budgets, n_keep):
    print(json.dumps(dict({"case": "attn", "workload": wl.name},
                          **attn_measure(R, synth, wl, dev, budgets, n_keep, args.layers,
                                         args.repeat))), flush=True)


def attn_measure(R, synth, wl, dev, budgets, n_keep, n_layers, repeat):
    """The scoring fused into the prefill attention of the window rows
    (ripple_compress_layers_attn) on the n_layers largest-budget layers in
    one call (each layer with its own inputs, above L2), beside
    ripple_compress_layers on the same inputs. Algorithmic bytes of the fused
    call: the compression's, plus V read in full and the fp32 outputs. The
    separate alternative would read the window rows' K and V once more (the
    prefill attention of those rows): `separate_read_ms` is that read at the
    measured copy bandwidth."""
    import torch
    L, B, Hq, Hkv, d, e = (wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim,
                           wl.elem_bytes)
    nl = max(1, min(n_layers, L))
    lay = sorted(range(L), key=lambda i: -budgets[i])[:nl]
    desc = R.layer_desc(B, Hq, Hkv, d, wl.seq_len, wl.window, wl.pool_kernel, "max",
                        wl.torch_dtype)
    outs = [(torch.empty(B, Hkv, n_keep[i], d, dtype=wl.torch_dtype, device=dev),
             torch.empty(B, Hkv, n_keep[i], d, dtype=wl.torch_dtype, device=dev),
             torch.empty(B * Hkv * n_keep[i], dtype=torch.int32, device=dev)) for i in lay]
    # every layer its own inputs: layers reading one K/V would share it in L2
    ins = [(synth.layer_window_queries(wl, i, dev), synth.layer_keys(wl, i, dev),
            synth.layer_values(wl, i, dev)) for i in lay]
    tabs = R.CompressTables([x[0] for x in ins], [x[1] for x in ins], [x[2] for x in ins],
                            [o[0] for o in outs], [o[1] for o in outs], [o[2] for o in outs])
    o_win = [torch.empty(B, Hq, wl.window, d, device=dev) for _ in lay]
    ws_a = torch.empty(R.ripple_compress_layers_attn_workspace_bytes(desc, nl), dtype=torch.uint8,
                       device=dev)
    ws_c = torch.empty(R.ripple_compress_layers_workspace_bytes(desc, nl), dtype=torch.uint8,
                       device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    bud = [budgets[i] for i in lay]
    comp_bytes = sum(B * Hkv * d * e * (wl.seq_len + 3 * n_keep[i]) + B * Hq * wl.window * d * e
                     for i in lay)
    attn_bytes = comp_bytes + nl * (B * Hkv * wl.seq_len * d * e + B * Hq * wl.window * d * 4)

    def timed(fn):
        ts = []
        for i in range(repeat + 2):
            a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b_.record()
            if i >= 2:
                ts.append((a, b_))
        torch.cuda.synchronize()
        return statistics.mean(a.elapsed_time(b) for a, b in ts)

    ms_a = timed(lambda: R.ripple_compress_layers_attn(desc, bud, tabs, o_win, ws_a,
                                                       dev_status=status))
    ms_c = timed(lambda: R.ripple_compress_layers(desc, bud, tabs, ws_c, dev_status=status))
    assert int(status.item()) == 0, int(status.item())
    hbm, src = measured_peaks()
    kv_bytes = nl * 2 * B * Hkv * wl.seq_len * d * e
    gbs = attn_bytes / (ms_a / 1e3) / 1e9
    return {
        "what": (f"compress {nl} layers with the window rows' attention output in one call "
                 f"(layers {lay}, each with its own inputs)"),
        "calls": repeat, "ms_per_call": round(ms_a, 5), "bytes_per_call": attn_bytes,
        "gbs": round(gbs, 1), "frac_hbm": round(gbs / hbm, 4),
        "compress_only_ms": round(ms_c, 5),
        "extra_ms_for_outputs": round(ms_a - ms_c, 5),
        "separate_read_ms": round(kv_bytes / (hbm * 1e9) * 1e3, 5),
        "peak_source": src}


def run_profile_case(args, R, synth, wl, dev):
    """The offline profiling kernels on the workload's shapes (Sec. 4.3):
    perturb = Eq. 6 on one layer's whole V cache (B, Hkv, T, d of the
    workload; the observation window protected), out of place;
    kl = Eq. 7 for n_layers perturbed runs (one per layer) against the
    reference, over a window of `window` positions and --vocab fp32 logits.
    Inputs exceed L2 (129 MB), so calls need no flush in between."""
    import torch
    B, Hkv, T, d, e = wl.batch, wl.n_kv_heads, wl.seq_len, wl.head_dim, wl.elem_bytes
    if args.case == "perturb":
        pb, pe, alpha = 0, T - wl.window, 0.05
        v = synth.layer_values(wl, 0, dev)
        eps = synth.perturb_draws(wl, 0, pe - pb, dev)
        out = torch.empty_like(v)
        call = lambda: R.ripple_perturb_values(v, eps, alpha, pb, pe, v_out=out)
        nbytes = 2 * B * Hkv * T * d * e + B * Hkv * (pe - pb) * d * 4
        what = (f"Eq. 6 on one layer's V cache [{B}][{Hkv}][{T}][{d}] {wl.dtype}, positions "
                f"[{pb}, {pe}) perturbed, out of place")
    else:
        n_sets, n_pos, vocab = wl.n_layers, wl.window, args.vocab
        p, q = synth.window_logits(wl.seed, n_sets, n_pos, vocab, torch.float32, dev)
        ws = torch.empty(R.ripple_window_kl_workspace_bytes(n_sets, n_pos, vocab),
                         dtype=torch.uint8, device=dev)
        d_out = torch.empty(n_sets, device=dev)
        kl_out = torch.empty(n_sets, n_pos, device=dev)
        call = lambda: R.ripple_window_kl(p, q, ws, d_out, kl_out)
        nbytes = (n_sets + 1) * n_pos * vocab * 4 + (n_sets * n_pos + n_sets) * 4
        what = (f"Eq. 7 for {n_sets} perturbed runs x {n_pos} window positions x {vocab} "
                f"fp32 logits")
    times = []
    for i in range(args.repeat + 2):
        a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        call()
        b_.record()
        if i >= 2:
            times.append((a, b_))
    torch.cuda.synchronize()
    ms = statistics.mean(a.elapsed_time(b) for a, b in times)
    hbm, src = measured_peaks()
    gbs = nbytes / (ms / 1e3) / 1e9
    print(json.dumps({"case": args.case, "workload": wl.name, "what": what, "calls": len(times),
                      "ms_per_call": round(ms, 5), "bytes_per_call": nbytes,
                      "gbs": round(gbs, 1), "frac_hbm": round(gbs / hbm, 4),
                      "peak_source": src}), flush=True)


def serving_loop_measure(R, synth, wl, dev, steps):
    """The per-layer serving shape (Sec. 4.1; Table 3's decode): every layer
    calls ripple_decode_attn on its own cache between stand-in projections
    (torch matmuls hidden -> q/k/v and attention output -> hidden; not the
    method), one step of all layers captured in a CUDA graph and replayed per
    token. Returns ms per token step of the whole loop, of the same graph
    without the projections (per-layer decode launches only) and of the
    all-layers decode launch on the same caches."""
    import torch

    from paper_2608_08684_gb300.serving import LayerDecodeLoop
    L, B, Hq, Hkv, d = wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim
    dt = wl.torch_dtype
    budgets = R.ripple_alloc_budgets(synth.sensitivity_profile(wl), wl.ratio, wl.gamma,
                                     wl.global_budget)
    n_keep = [R.ripple_keep_count(b, wl.seq_len, wl.window) for b in budgets]
    warm = 3
    caps = [n + 2 * (steps + warm) + 2 for n in n_keep]
    kc, vc = zip(*[synth.decode_caches(wl, l, caps[l], dev) for l in range(L)])
    kc, vc = list(kc), list(vc)
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    hid = Hq * d
    h = torch.randn(B, hid, generator=g, device=dev).to(dt)
    wqkv = [(torch.randn(hid, (Hq + 2 * Hkv) * d, generator=g, device=dev) / hid ** 0.5).to(dt)
            for _ in range(L)]
    wo = [(torch.randn(hid, hid, generator=g, device=dev) / hid ** 0.5).to(dt) for _ in range(L)]
    qb = torch.zeros(1, B, Hq, d, dtype=dt, device=dev)
    kb = torch.zeros(1, B, Hkv, d, dtype=dt, device=dev)
    vb = torch.zeros(1, B, Hkv, d, dtype=dt, device=dev)

    def before(l):
        hn = h.float()
        x = (hn * torch.rsqrt(hn.square().mean(-1, keepdim=True) + 1e-6)).to(dt) @ wqkv[l]
        qb.copy_(x[:, :Hq * d].reshape(1, B, Hq, d))
        kb.copy_(x[:, Hq * d:(Hq + Hkv) * d].reshape(1, B, Hkv, d))
        vb.copy_(x[:, (Hq + Hkv) * d:].reshape(1, B, Hkv, d))
        return qb, kb, vb

    def after(l, out):
        h.add_(out.reshape(B, hid).to(dt) @ wo[l])

    def timed(fn, n):
        for _ in range(warm):
            fn()
        torch.cuda.synchronize()
        a, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(n):
            fn()
        b_.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b_) / n

    lens = torch.tensor(n_keep, dtype=torch.int32, device=dev)
    full = LayerDecodeLoop(kc, vc, lens, Hq, before, after)
    full.issue_step()
    full.capture()
    ms_full = timed(full.replay, steps)
    lens.copy_(torch.tensor(n_keep, dtype=torch.int32, device=dev))
    attn = LayerDecodeLoop(kc, vc, lens, Hq, lambda l: (qb, kb, vb), lambda l, o: None)
    attn.issue_step()
    attn.capture()
    ms_attn = timed(attn.replay, steps)
    assert int(full.status.item()) == 0 and int(attn.status.item()) == 0
    # the all-layers launch on the same caches (one decode kernel per step)
    lens.copy_(torch.tensor(n_keep, dtype=torch.int32, device=dev))
    ddesc = R.decode_desc(L, B, Hq, Hkv, d, dt)
    tables = R.DecodeTables(kc, vc)
    dws = torch.empty(R.ripple_decode_workspace_bytes(ddesc, caps), dtype=torch.uint8, device=dev)
    q, kn, vn = synth.decode_inputs(wl, 0, dev)
    out = torch.empty(L, B, Hq, d, device=dev)
    ms_one = timed(lambda: R.ripple_decode_attn(ddesc, q, kn, vn, tables, lens, out, dws), steps)
    return {"steps": steps, "ms_per_token_step": round(ms_full, 4),
            "tokens_per_s": round(B / (ms_full / 1e3), 1),
            "per_layer_decode_launches_ms_per_step": round(ms_attn, 4),
            "all_layers_one_launch_ms_per_step": round(ms_one, 4),
            "what": (f"{L} layers x (stand-in q/k/v projection, single-layer ripple_decode_attn "
                     f"appending, stand-in output projection) per token, CUDA graph replayed "
                     f"{steps} times; caches at the RippleKV sizes ({min(n_keep)}..{max(n_keep)} "
                     f"rows)")}


def profile_traffic(profile, sources, alg_bytes):
    """DRAM traffic (read + write bytes) of one launch from a committed ncu
    summary under profiles/, scaled from the captured launch to this one by
    algorithmic bytes. None when the kernel's sources changed since the
    capture (their hash differs) or the summary is missing."""
    import hashlib
    path = os.path.join(ROOT, "profiles", profile)
    try:
        fields = {}
        for line in open(path):
            if ":" in line and not line.startswith(("|", "#", " ")):
                k, v = line.split(":", 1)
                fields[k.strip()] = v.strip()
        h = hashlib.sha256()
        for s in sources:
            with open(os.path.join(ROOT, "paper_2608_08684_gb300", "csrc", s), "rb") as f:
                h.update(f.read())
        if h.hexdigest()[:16] != fields["source_sha256"]:
            return None
        traffic = float(fields["traffic_bytes_per_launch"])
        captured = float(fields["algorithmic_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        return None
    return round(traffic * alg_bytes / captured)


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return HBM_FALLBACK_GBS, "fallback"


# ----------------------------------------------------------------- clocks


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    def __init__(self, gpu_index: int):
        self.gpu_index = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active")
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={q}", "--format=csv,noheader,nounits", "-lms", "100",
                 "-i", str(self.gpu_index)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons, power = [], None, set(), []
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 5:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
                power.append(float(parts[3]))
                bits = int(parts[4], 16)
            except ValueError:
                continue
            for b, name in REASON_BITS.items():
                if bits & b and name != "gpu_idle":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm), "power_w_max": max(power) if power else None}


# ----------------------------------------------------------------- workload state


class Serving:
    """Device-resident inputs, outputs and workspaces of one workload."""

    def __init__(self, R, synth, wl, device):
        import torch
        self.R, self.wl, self.dev = R, wl, device
        L, B, Hq, Hkv, d = wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim
        self.sens = synth.sensitivity_profile(wl)
        self.budgets = R.ripple_alloc_budgets(self.sens, wl.ratio, wl.gamma, wl.global_budget)
        self.n_keep = [R.ripple_keep_count(b, wl.seq_len, wl.window) for b in self.budgets]
        self.caps = [n + wl.decode_steps for n in self.n_keep]
        self.q_win, self.k, self.v = [], [], []
        for layer in range(L):
            self.q_win.append(synth.layer_window_queries(wl, layer, device))
            self.k.append(synth.layer_keys(wl, layer, device))
            self.v.append(synth.layer_values(wl, layer, device))
        self.desc = R.layer_desc(B, Hq, Hkv, d, wl.seq_len, wl.window, wl.pool_kernel, "max",
                                 wl.torch_dtype)
        # one call compresses every layer (ripple_compress_layers)
        self.ws = torch.empty(R.ripple_compress_layers_workspace_bytes(self.desc, L),
                              dtype=torch.uint8, device=device)
        self.k_out = [torch.zeros(B, Hkv, c, d, dtype=wl.torch_dtype, device=device)
                      for c in self.caps]
        self.v_out = [torch.zeros_like(t) for t in self.k_out]
        self.idx = [torch.empty(B * Hkv * n, dtype=torch.int32, device=device)
                    for n in self.n_keep]
        self.ctables = R.CompressTables(self.q_win, self.k, self.v, self.k_out, self.v_out,
                                        self.idx)
        self.status = torch.zeros(1, dtype=torch.int32, device=device)
        # every decode step's inputs in one tensor per kind (dq[t] is a view),
        # so that the end-to-end run copies them in three copies
        steps = [synth.decode_inputs(wl, t, device) for t in range(wl.decode_steps)]
        self.dq_all, self.dk_all, self.dv_all = (torch.stack([x[i] for x in steps])
                                                 for i in range(3))
        del steps
        self.dq, self.dk, self.dv = (list(x.unbind(0))
                                     for x in (self.dq_all, self.dk_all, self.dv_all))
        self.ddesc = R.decode_desc(L, B, Hq, Hkv, d, wl.torch_dtype)
        self.tables = R.DecodeTables(self.k_out, self.v_out)
        self.dws = torch.empty(R.ripple_decode_workspace_bytes(self.ddesc, self.caps),
                               dtype=torch.uint8, device=device)
        self.lens0 = torch.tensor(self.n_keep, dtype=torch.int32, device=device)
        self.lens = self.lens0.clone()
        self.out = torch.empty(wl.decode_steps, L, B, Hq, d, dtype=torch.float32, device=device)

    def step(self, timers=None):
        """One pass of the whole path; timers = (compress_events, decode_events) or None."""
        import torch
        R, wl = self.R, self.wl
        budgets = R.ripple_alloc_budgets(self.sens, wl.ratio, wl.gamma, wl.global_budget)
        assert budgets == self.budgets
        ev = (lambda: torch.cuda.Event(enable_timing=True)) if timers else None
        if timers:
            c0 = ev()
            c0.record()
        n = R.ripple_compress_layers(self.desc, budgets, self.ctables, self.ws,
                                     dev_status=self.status)
        assert n == self.n_keep
        if timers:
            c1 = ev()
            c1.record()
            timers[0].append((c0, c1))
        self.lens.copy_(self.lens0)
        # the decode steps run back to back (each launch may overlap the
        # previous one's tail); one event pair brackets all of them
        if timers:
            d0 = ev()
            d0.record()
        for t in range(wl.decode_steps):
            R.ripple_decode_attn(self.ddesc, self.dq[t], self.dk[t], self.dv[t], self.tables,
                                 self.lens, self.out[t], self.dws, dev_status=self.status)
        if timers:
            d1 = ev()
            d1.record()
            timers[1].append((d0, d1))

    # algorithmic bytes (what the method must move)
    def compress_bytes(self):
        wl, e = self.wl, self.wl.elem_bytes
        tot = 0
        for n in self.n_keep:
            tot += wl.batch * wl.n_kv_heads * wl.head_dim * e * (wl.seq_len + 3 * n)
            tot += wl.batch * wl.n_q_heads * wl.window * wl.head_dim * e
        return tot

    def decode_bytes_per_step(self):
        """Average over the decode steps: K/V rows read (retained + appended +
        the new row), queries read, outputs written, new rows read and appended."""
        wl, e = self.wl, self.wl.elem_bytes
        L, B, Hq, Hkv, d = wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim
        tot = 0
        for t in range(wl.decode_steps):
            for n in self.n_keep:
                tot += B * Hkv * (n + t + 1) * d * e * 2
            tot += L * B * Hq * d * (e + 4) + L * B * Hkv * d * e * 4
        return tot / wl.decode_steps


def measure_workloads(R, synth, dev, names, reps):
    """The serving step on other workloads (each generated, timed and freed in
    turn): compression of all layers and decode steps, with their fractions of
    the measured HBM bandwidth; for compression also the tensor-pipe fraction
    of the window-query contraction (two passes, 2 * G*w * T * d flops per
    unit and pass) against the measured sustained bf16 peak, and for decode the
    fp32 FMA fraction (q.k and p.v: 2 * d FMAs per cached row and query head)
    against the peak derived from the SM count, 128 FMA lanes per SM and the
    maximum SM clock."""
    import torch
    hbm, _ = measured_peaks()
    tensor_peak = measured_peak("bf16_tflops_sustained", 1700.0)
    props = torch.cuda.get_device_properties(dev)
    fma_peak = props.multi_processor_count * 128 * 2 * measured_peak("sm_max_mhz", 2070.0) * 1e6 / 1e12
    res = {}
    for name in names:
        wl = synth.WORKLOADS[name]
        st = Serving(R, synth, wl, dev)
        for _ in range(2):
            st.step()
        torch.cuda.synchronize()
        timers = ([], [])
        for _ in range(reps):
            st.step(timers)
        torch.cuda.synchronize()
        assert int(st.status.item()) == 0
        comp = statistics.mean(elapsed_ms(timers[0]))
        dec = statistics.mean(elapsed_ms(timers[1])) / wl.decode_steps
        R_rows, units = wl.group * wl.window, wl.batch * wl.n_kv_heads
        flops = sum(4.0 * R_rows * wl.seq_len * wl.head_dim * units
                    for n in st.n_keep if n < wl.seq_len)
        fmas = sum(units * (n + t + 1) * wl.group * 2 * wl.head_dim
                   for t in range(wl.decode_steps) for n in st.n_keep) / wl.decode_steps
        cg = st.compress_bytes() / (comp / 1e3) / 1e9
        dg = st.decode_bytes_per_step() / (dec / 1e3) / 1e9
        res[name] = {"workload": wl.name, "dtype": wl.dtype,
                     "compress_ms": round(comp, 4), "compress_gbs": round(cg, 1),
                     "compress_frac_hbm": round(cg / hbm, 4),
                     "compress_tokens_per_s": round(wl.batch * wl.seq_len / (comp / 1e3), 1),
                     "compress_tensor_tflops": round(flops / (comp / 1e3) / 1e12, 1),
                     "compress_frac_tensor_sustained": round(flops / (comp / 1e3) / 1e12 / tensor_peak, 4),
                     "decode_ms_per_step": round(dec, 5), "decode_gbs": round(dg, 1),
                     "decode_frac_hbm": round(dg / hbm, 4),
                     "decode_fma_tflops": round(2 * fmas / (dec / 1e3) / 1e12, 2),
                     "decode_frac_fma_peak": round(2 * fmas / (dec / 1e3) / 1e12 / fma_peak, 4),
                     "step_ms": round(comp + dec * wl.decode_steps, 3),
                     "reps": reps}
        del st
        torch.cuda.empty_cache()
    res["peaks"] = {"hbm_gbs": hbm, "bf16_tflops_sustained": tensor_peak,
                    "fp32_fma_tflops_derived": round(fma_peak, 1)}
    return res


def measured_peak(key, fallback):
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)[key])
    except Exception:
        return fallback


def workload_config(wl, world, budgets):
    """The `config` object of a bench line (both arms report the same one)."""
    return {"workload": wl.name, "layers": wl.n_layers, "batch": wl.batch,
            "q_heads": wl.n_q_heads, "kv_heads": wl.n_kv_heads, "head_dim": wl.head_dim,
            "seq_len": wl.seq_len, "window": wl.window, "pool_kernel": wl.pool_kernel,
            "ratio": wl.ratio, "avg_budget": wl.avg_budget, "decode_steps": wl.decode_steps,
            "budgets": list(budgets), "parallelism": f"replicas{world}",
            "l2": "inputs larger than L2 (K+V per layer %.0f MB), no flush"
                  % (2 * wl.batch * wl.n_kv_heads * wl.seq_len * wl.head_dim * wl.elem_bytes / 1e6)}


def elapsed_ms(pairs):
    return [a.elapsed_time(b) for a, b in pairs]


def replica_workload(wl, rank):
    """Rank r of a multi-GPU run serves its own independent batch (replicas:
    the path has no exchange step), seeded apart from the other ranks."""
    return wl.replace(seed=wl.seed + 1000 * rank) if rank else wl


def max_over_ranks(ms, world, device):
    """The timed region's length as the slowest rank saw it."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    tt = torch.tensor([ms], device=device, dtype=torch.float64)
    dist.all_reduce(tt, op=dist.ReduceOp.MAX)
    return float(tt.item())


def job_throughput(total_ms, steps, tokens_per_rank, world):
    """(ms per step, whole-job tokens/s): every rank processed its own batch
    within the max-over-ranks time."""
    ms_per_step = total_ms / steps
    return ms_per_step, tokens_per_rank * world / (ms_per_step / 1e3)


def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    from paper_2608_08684_gb300 import build as _build
    from paper_2608_08684_gb300 import synth

    device = torch.device("cuda", local_rank)
    torch.cuda.set_device(device)
    if world > 1:
        dist.init_process_group("nccl", device_id=device)
    if rank == 0:
        _build.build_library()
    if world > 1:
        dist.barrier()
    from paper_2608_08684_gb300 import ripple as R

    wl = synth.WORKLOADS[args.workload]
    # independent replicas: every rank serves its own batch (weak scaling)
    wl = replica_workload(wl, rank)
    st = Serving(R, synth, wl, device)
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    for _ in range(args.warmup):
        st.step()
    barrier()
    assert int(st.status.item()) == 0, f"device status {int(st.status.item())}"
    launches0 = R.ripple_kernel_launches()
    timers = ([], [])
    gpu_index = int(os.environ.get("CUDA_VISIBLE_DEVICES", str(local_rank)).split(",")[0]) \
        if os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")[0].isdigit() else local_rank
    with ClockSampler(gpu_index) as clocks:
        barrier()
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        for _ in range(args.steps):
            st.step(timers)
        t1.record()
        barrier()
    launches = R.ripple_kernel_launches() - launches0
    assert int(st.status.item()) == 0
    total_ms = max_over_ranks(t0.elapsed_time(t1), world, device)
    ms_per_step, value = job_throughput(total_ms, args.steps, wl.batch * wl.seq_len, world)
    tokens = wl.batch * wl.seq_len * world

    comp_ms = elapsed_ms(timers[0])
    dec_ms = [ms / wl.decode_steps for ms in elapsed_ms(timers[1])]  # per decode launch
    hbm, hbm_src = measured_peaks()
    comp_avg = statistics.mean(comp_ms)
    dec_avg = statistics.mean(dec_ms)
    comp_gbs = st.compress_bytes() / (comp_avg / 1e3) / 1e9
    dec_gbs = st.decode_bytes_per_step() / (dec_avg / 1e3) / 1e9
    comp_total = comp_avg
    dec_total = dec_avg * wl.decode_steps
    dec_traffic = profile_traffic("decode_kernel_llama3-8b_B4_T32768.md",
                                  ["decode.cu", "decode.cuh", "common.cuh"],
                                  st.decode_bytes_per_step()) \
        if wl.name.startswith("llama3-8b-32L-32q8kv-d128-B4-T32768") else None
    roof_dec = {"bound": "hbm", "achieved": round(dec_gbs, 1), "peak": hbm, "unit": "GB/s",
                "frac": round(dec_gbs / hbm, 4), "traffic": dec_traffic,
                "traffic_source": ("ncu dram bytes of the first decode step "
                                   "(profiles/decode_kernel_llama3-8b_B4_T32768.md), scaled "
                                   "by algorithmic bytes") if dec_traffic else None,
                "kernel": "decode_kernel (ripple_decode_attn, one launch per step)",
                "bytes_per_launch": round(st.decode_bytes_per_step()),
                "ms_per_launch": round(dec_avg, 5), "peak_source": hbm_src}
    comp_traffic = profile_traffic("compress_kernels_llama3-8b_B4_T32768_8layers.md",
                                   ["score_tc1.cu", "select.cu", "tc_ptx.cuh", "common.cuh"],
                                   st.compress_bytes()) \
        if wl.name.startswith("llama3-8b-32L-32q8kv-d128-B4-T32768") else None
    roof_comp = {"bound": "hbm", "achieved": round(comp_gbs, 1), "peak": hbm, "unit": "GB/s",
                 "frac": round(comp_gbs / hbm, 4), "traffic": comp_traffic,
                 "traffic_source": ("ncu dram bytes of the two kernels on an 8-layer "
                                    "ripple_compress_layers call (profiles/compress_kernels_"
                                    "llama3-8b_B4_T32768_8layers.md), scaled to all layers by "
                                    "algorithmic bytes")
                 if comp_traffic else None,
                 "kernel": ("score_tc1_kernel + select_unit_kernel (with the gather) "
                            "(ripple_compress_layers, all layers in two launches)"),
                 "bytes_per_launch": round(st.compress_bytes()),
                 "ms_per_launch": round(comp_avg, 4), "peak_source": hbm_src}
    dominant = roof_dec if dec_total >= comp_total else roof_comp

    e2e = None
    if not args.no_e2e:
        e2e = measure_e2e(st, args, torch, tokens // world * world)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(st, args.cpu_seconds)
    budgets = st.budgets
    others = serving = fused = None
    if rank == 0 and world == 1 and not args.no_workloads:
        # the other workloads and the per-layer serving loop, after the
        # headline workload's buffers are freed
        del st, timers
        torch.cuda.empty_cache()
        with ClockSampler(gpu_index) as oclocks:
            others = measure_workloads(R, synth, device,
                                       [n for n in synth.WORKLOADS if n != args.workload], 3)
            serving = serving_loop_measure(R, synth, wl, device, 32)
            fused = attn_measure(R, synth, wl, device, budgets,
                                 [R.ripple_keep_count(b, wl.seq_len, wl.window) for b in budgets],
                                 wl.n_layers, 3) if wl.dtype == "bf16" and wl.head_dim == 128 \
                and wl.group * wl.window == 128 else None
        others["clocks"] = oclocks.summary()
    if rank != 0:
        return
    line = {
        "metric": METRIC,
        "value": round(value, 1), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": workload_config(wl, world, budgets),
        "compress": {"tokens_per_s": round(tokens / world / (comp_avg / 1e3), 1),
                     "ms": round(comp_avg, 4), "gbs": round(comp_gbs, 1),
                     "frac_hbm": round(comp_gbs / hbm, 4),
                     "frac_8tbs_spec": round(comp_gbs / 8000.0, 4)},
        "decode_attn": {"gbs": round(dec_gbs, 1), "ms_per_step": round(dec_avg, 5),
                        "frac_hbm": round(dec_gbs / hbm, 4),
                        "frac_8tbs_spec": round(dec_gbs / 8000.0, 4)},
        "roofline": dominant,
        "roofline_compress": roof_comp,
        "roofline_decode": roof_dec,
        "gpu_launches": launches,
        "clocks": clocks.summary(),
    }
    if e2e:
        line["e2e"] = e2e
    if others:
        line["workloads"] = others
        line["serving_loop"] = serving
        if fused:
            line["compress_attn"] = fused
    if cpu:
        line["cpu_baseline"] = cpu
    print(json.dumps(line), flush=True)


def measure_e2e(st, args, torch, tokens, group=8):
    """Same metric through the C ABI from pinned host buffers: every step copies
    the layer inputs and decode inputs host->device and reads the decode
    outputs back, inside the timed region. The copies run on a second stream
    in groups of `group` layers; each group is compressed
    (ripple_compress_layers) as soon as it has landed, while the next one is
    copied, and the decode outputs go back in four parts behind the decode
    steps."""
    wl, R = st.wl, st.R
    L = wl.n_layers

    def pin(t):
        h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        h.copy_(t)
        return h

    hq = [pin(t) for t in st.q_win]
    hk = [pin(t) for t in st.k]
    hv = [pin(t) for t in st.v]
    hd = [pin(t) for t in (st.dq_all, st.dk_all, st.dv_all)]
    hout = torch.empty(st.out.shape, dtype=st.out.dtype).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in hq + hk + hv + hd)
    d2h = hout.numel() * hout.element_size()
    groups = [(g, min(L, g + group)) for g in range(0, L, group)]
    tables = [R.CompressTables(st.q_win[a:b], st.k[a:b], st.v[a:b], st.k_out[a:b],
                               st.v_out[a:b], st.idx[a:b]) for a, b in groups]
    main, side = torch.cuda.current_stream(), torch.cuda.Stream()
    landed = [torch.cuda.Event() for _ in groups]
    dec_in, start = torch.cuda.Event(), torch.cuda.Event()
    parts = [(t, min(wl.decode_steps, t + (wl.decode_steps + 3) // 4))
             for t in range(0, wl.decode_steps, (wl.decode_steps + 3) // 4)]
    done = [torch.cuda.Event() for _ in parts]

    def step():
        start.record(main)
        side.wait_event(start)  # the previous step is done with the inputs
        with torch.cuda.stream(side):
            st.dq_all.copy_(hd[0], non_blocking=True)
            st.dk_all.copy_(hd[1], non_blocking=True)
            st.dv_all.copy_(hd[2], non_blocking=True)
            dec_in.record(side)
            for (a, b), ev in zip(groups, landed):
                for layer in range(a, b):
                    st.q_win[layer].copy_(hq[layer], non_blocking=True)
                    st.k[layer].copy_(hk[layer], non_blocking=True)
                    st.v[layer].copy_(hv[layer], non_blocking=True)
                ev.record(side)
        for (a, b), ev, tab in zip(groups, landed, tables):
            main.wait_event(ev)
            n = R.ripple_compress_layers(st.desc, st.budgets[a:b], tab, st.ws,
                                         dev_status=st.status)
            assert n == st.n_keep[a:b]
        main.wait_event(dec_in)
        st.lens.copy_(st.lens0)
        for (t0, t1), ev in zip(parts, done):
            for t in range(t0, t1):
                R.ripple_decode_attn(st.ddesc, st.dq[t], st.dk[t], st.dv[t], st.tables, st.lens,
                                     st.out[t], st.dws, dev_status=st.status)
            ev.record(main)
            side.wait_event(ev)
            with torch.cuda.stream(side):
                hout[t0:t1].copy_(st.out[t0:t1], non_blocking=True)
        main.wait_stream(side)

    # freshly pinned buffers copy at a fraction of the link's rate for their
    # first one or two uses (measured: 124-178 ms, then 83 ms for the same
    # 17.4 GB), so three untimed steps come first
    for _ in range(3):
        step()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(args.e2e_steps):
        step()
    t1.record()
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / args.e2e_steps
    return {"value": round(tokens / (ms / 1e3), 1), "unit": "tokens/s", "ms_per_step": round(ms, 3),
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": args.e2e_steps,
            "warmup_steps": 3,
            "overlap": f"host->device copies on a second stream, compression per {group} layers "
                       "as they land, outputs back in four parts behind the decode steps"}


# ----------------------------------------------------------------- CPU oracle


# ----------------------------------------------------------------- CPU oracle
#
# The oracle is timed on a bounded sample of the workload by a pool of worker
# processes (spawned, one BLAS/torch thread each, one per host core); each
# worker regenerates its layer's seeded inputs on the host, then times whole
# compression units (compress_unit) and decode steps of single groups
# (decode_attention) until its time budget is spent. The full step's time is
# extrapolated from the pool's aggregate rates: a reported baseline only.


def _oracle_worker_init():
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[var] = "1"


def _oracle_worker(task):
    """One sampling task in a worker process: ("compress", workload fields,
    layer, budget, [(b, h), ...], seconds) or ("decode", workload fields,
    layer, n_keep, steps, seconds). Returns (units or group-steps done, compute
    seconds)."""
    import numpy as np
    import torch

    from oracle import ripple_oracle as O
    from paper_2608_08684_gb300 import synth
    torch.set_num_threads(1)
    kind, fields, layer = task[0], task[1], task[2]
    wl = synth.Workload(**fields)
    G, scale = wl.group, 1.0 / math.sqrt(wl.head_dim)
    if kind == "compress":
        budget, units, seconds = task[3], task[4], task[5]
        q = synth.layer_window_queries(wl, layer)
        k = synth.layer_keys(wl, layer)
        v = synth.layer_values(wl, layer)
        done, spent = 0, 0.0
        for b, h in units:
            if spent >= seconds:
                break
            qu = synth.to_f64(q[b, h * G:(h + 1) * G])
            ku, vu = synth.to_f64(k[b, h]), synth.to_f64(v[b, h])
            t = time.perf_counter()
            O.compress_unit(qu, ku, vu, budget, wl.window, scale, wl.pool_kernel)
            spent += time.perf_counter() - t
            done += 1
        return done, spent
    n_keep, steps, seconds = task[3], task[4], task[5]
    one = wl.replace(batch=1, n_kv_heads=1, n_q_heads=G)
    kc, vc = synth.decode_caches(one, layer, n_keep)
    rows_k, rows_v = synth.to_f64(kc[0, 0]), synth.to_f64(vc[0, 0])
    done, spent = 0, 0.0
    for s in range(steps):
        if spent >= seconds:
            break
        q, kn, vn = synth.decode_inputs(one, s, layers=[layer])
        qq, kk, vv = synth.to_f64(q[0, 0]), synth.to_f64(kn[0, 0, 0]), synth.to_f64(vn[0, 0, 0])
        t = time.perf_counter()
        rows_k = np.vstack([rows_k, kk[None]])
        rows_v = np.vstack([rows_v, vv[None]])
        O.decode_attention(qq, rows_k, rows_v, scale)
        spent += time.perf_counter() - t
        done += 1
    return done, spent


def oracle_step_time(wl, budgets, n_keep, target_s, layers=None, workers=None):
    """Times the oracle on a bounded sample with a pool of worker processes
    and extrapolates to one full step. Returns a dict with the step seconds,
    the worker count, the sampled fraction and a description."""
    import multiprocessing as mp
    workers = workers or os.cpu_count() or 1
    layers = list(range(wl.n_layers)) if layers is None else list(layers)
    fields = dict(wl.__dict__)
    units_all = [(b, h) for b in range(wl.batch) for h in range(wl.n_kv_heads)]
    # compression: one task per worker, round robin over the sampled layers,
    # each task taking a strided share of its layer's units
    per_layer = max(1, workers // len(layers))
    ctasks = []
    for i in range(max(workers, len(layers))):
        layer = layers[i % len(layers)]
        share = units_all[(i // len(layers)) % per_layer::per_layer]
        ctasks.append(("compress", fields, layer, budgets[layer], share, 0.75 * target_s))
    steps = min(16, wl.decode_steps)
    dtasks = [("decode", fields, layer, n_keep[layer], steps, 0.25 * target_s)
              for layer in layers[:workers]]
    t0 = time.perf_counter()
    with mp.get_context("spawn").Pool(workers, initializer=_oracle_worker_init) as pool:
        cres = pool.map(_oracle_worker, ctasks, chunksize=1)
        dres = pool.map(_oracle_worker, dtasks, chunksize=1)
    wall = time.perf_counter() - t0
    # aggregate rates: every worker runs in parallel with the others
    c_rate = sum(d / s for d, s in cres if s > 0)
    d_rate = sum(d / s for d, s in dres if s > 0)
    units_total = wl.n_layers * wl.batch * wl.n_kv_heads
    group_steps = wl.n_layers * wl.batch * wl.n_kv_heads * wl.decode_steps
    step_s = units_total / c_rate + group_steps / d_rate
    n_units = sum(d for d, _ in cres)
    n_dec = sum(d for d, _ in dres)
    return {"step_s": step_s, "workers": workers, "wall_s": wall,
            "sample_fraction": (n_units + n_dec) / (units_total + group_steps),
            "sample": (f"{n_units} compression units (T={wl.seq_len}, {len(layers)} layers "
                       f"{layers if len(layers) <= 8 else '(evenly spaced)'}) "
                       f"and {n_dec} decode group-steps timed by {workers} worker processes "
                       f"(one thread each); extrapolated to {units_total} units and "
                       f"{group_steps} group-steps by the pool's aggregate rates")}


def cpu_baseline(st, target_s):
    wl = st.wl
    # one task per worker: evenly spaced layers, at most one per worker
    workers = os.cpu_count() or 1
    n = min(workers, wl.n_layers)
    layers = sorted({round(i * (wl.n_layers - 1) / max(1, n - 1)) for i in range(n)})
    r = oracle_step_time(wl, st.budgets, st.n_keep, target_s, layers=layers, workers=workers)
    return {"value": round(wl.batch * wl.seq_len / r["step_s"], 2), "unit": "tokens/s",
            "cores": r["workers"], "kind": "oracle", "sample": r["sample"],
            "extrapolated": True, "sample_fraction": round(r["sample_fraction"], 5),
            "wall_s": round(r["wall_s"], 1),
            "step_seconds_extrapolated": round(r["step_s"], 2)}


def run_reference(args, rank, world):
    """Reference arm: the CPU oracle, timed on this host's cores (a pool of
    worker processes), each step a bounded sample of the workload extrapolated
    to a full step."""
    if rank != 0:
        return
    from oracle import ripple_oracle as O
    from paper_2608_08684_gb300 import synth
    wl = synth.WORKLOADS[args.workload]
    budgets = O.alloc_budgets(synth.sensitivity_profile(wl), wl.ratio, wl.gamma,
                              wl.global_budget)
    n_keep = [O.keep_count(b, wl.seq_len, wl.window) for b in budgets]
    # four sampled layers: largest and smallest budget, two in between
    by_budget = sorted(range(wl.n_layers), key=lambda i: budgets[i])
    sample_layers = sorted({by_budget[-1], by_budget[0], by_budget[len(by_budget) // 3],
                            by_budget[2 * len(by_budget) // 3]})
    per_step = max(2.0, min(args.cpu_seconds, 120.0 / max(1, args.steps + args.warmup)))
    times, r = [], None
    for i in range(args.warmup + args.steps):
        r = oracle_step_time(wl, budgets, n_keep, per_step, layers=sample_layers)
        if i >= args.warmup:
            times.append(r["step_s"])
    step_s = statistics.mean(times)
    value = wl.batch * wl.seq_len / step_s
    line = {"metric": METRIC,
            "value": round(value, 2), "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(step_s * 1e3, 1),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": workload_config(wl, world, budgets),
            "cpu_baseline": {"value": round(value, 2), "unit": "tokens/s", "cores": r["workers"],
                             "kind": "oracle", "sample": r["sample"], "extrapolated": True,
                             "sample_fraction": round(r["sample_fraction"], 5)},
            "e2e": {"value": round(value, 2), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
            "note": ("each step times a bounded sample of the workload and reports the "
                     "extrapolated time of a full step; ms_per_step is that extrapolation, "
                     "not the wall time of the sample")}
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", str(args.gpus if args.gpus == 1 else 1)))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.case:
        run_case(args)
    elif args.impl == "reference":
        run_reference(args, rank, world)
    else:
        run_ours(args, rank, world, local_rank)


if __name__ == "__main__":
    main()
