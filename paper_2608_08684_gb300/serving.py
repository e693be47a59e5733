"""Per-layer decode loop over the ragged compressed caches, captured in a CUDA graph.

Sec. 4.1: during decoding each new query attends to the cached states, layer
after layer; the paper's end-to-end decode throughput (Table 3) is measured
in that shape. Here every layer calls ripple_decode_attn on its own cache
(one layer per call, appending the step's key/value row), with the caller's
per-layer work around each call (the projections that produce the layer's
query/key/value rows and consume its attention output). One decode step of
all layers is captured once in a CUDA graph and replayed per generated token.

Orchestration only: each layer's attention runs in libripple's decode kernel;
the per-layer callables belong to the caller. The graph reads each layer's
cache length from device memory, and the kernel advances it, so replays keep
appending.
"""
from __future__ import annotations

import torch

from . import ripple as R


class LayerDecodeLoop:
    """One decode step of L layers as L single-layer ripple_decode_attn calls.

    k_caches, v_caches: per layer [B][Hkv][cap_l][d] device tensors (the
        compressed caches with room for the appended rows).
    lens: device int32 [L], rows in use per layer; advanced by every step.
    before(l): returns (q [1][B][Hq][d], k_new [1][B][Hkv][d],
        v_new [1][B][Hkv][d]) contiguous device tensors of layer l's new token
        (in the caches' dtype); called while the step is issued (and captured).
    after(l, out): consumes layer l's attention output out [1][B][Hq][d] fp32.
    """

    def __init__(self, k_caches, v_caches, lens, n_q_heads, before, after, scale=0.0):
        self.L = len(k_caches)
        B, Hkv, _, d = k_caches[0].shape
        self.before, self.after = before, after
        self.lens = lens
        self.descs = [R.decode_desc(1, B, n_q_heads, Hkv, d, k_caches[0].dtype, scale)
                      for _ in range(self.L)]
        self.tables = [R.DecodeTables([k], [v]) for k, v in zip(k_caches, v_caches)]
        ws = max(R.ripple_decode_workspace_bytes(self.descs[l], [k_caches[l].shape[-2]])
                 for l in range(self.L))
        dev = k_caches[0].device
        # calls are ordered on one stream, so every layer shares the workspace
        self.ws = torch.empty(ws, dtype=torch.uint8, device=dev)
        self.out = [torch.empty(1, B, n_q_heads, d, dtype=torch.float32, device=dev)
                    for _ in range(self.L)]
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.graph = None

    def issue_step(self):
        """Enqueue one decode step of every layer on the current stream."""
        for l in range(self.L):
            q, kn, vn = self.before(l)
            R.ripple_decode_attn(self.descs[l], q, kn, vn, self.tables[l], self.lens[l:l + 1],
                                 self.out[l], self.ws, dev_status=self.status)
            self.after(l, self.out[l])

    def capture(self):
        """Capture one step in a CUDA graph. Run issue_step() once outside the
        capture first (the library's first call on a device sets the decode
        kernel's attributes); that step appends like any other."""
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            self.issue_step()
        return self.graph

    def replay(self):
        self.graph.replay()
