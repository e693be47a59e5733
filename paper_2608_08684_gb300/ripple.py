"""Python binding of libripple.so (the C ABI declared in include/ripple.h).

Argument marshalling only: every function here passes raw pointers, sizes and
the current CUDA stream to the entry point of the same name, and raises
RippleError on a non-zero status. All computation happens in the library's
kernels (or, for ripple_alloc_budgets, in its host C code). Importing this
module fails loudly if the library has not been built.
"""
from __future__ import annotations

import ctypes
import os

import torch

# RIPPLE_CHECKED=1 selects the bounds-checked build of the same library.
CHECKED = os.environ.get("RIPPLE_CHECKED", "0") == "1"
LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)),
                        "libripple_checked.so" if CHECKED else "libripple.so")
if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is not built: call paper_2608_08684_gb300.build."
                      f"build_library(checked={CHECKED})")
_lib = ctypes.CDLL(LIB_PATH)

F32, BF16 = 0, 1
POOL_MAX, POOL_AVG, POOL_NONE = 0, 1, 2
OK, EINVAL, EWORKSPACE, EFULL, ECUDA, ETIMEOUT, EBOUNDS, ENOMEM = range(8)
MAX_LAYERS = 128
COMPRESS_MAX_LAYERS = 80
_POOLS = {"max": POOL_MAX, "avg": POOL_AVG, "none": POOL_NONE}
_DTYPES = {torch.float32: F32, torch.bfloat16: BF16}


class RippleError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


class LayerDesc(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("seq_len", ctypes.c_int32), ("window", ctypes.c_int32),
                ("pool_kernel", ctypes.c_int32), ("pool_type", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("scale", ctypes.c_float)]


class DecodeDesc(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("batch", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("scale", ctypes.c_float)]


class CacheDesc(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("seq_len", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("dtype", ctypes.c_int32)]


_p = ctypes.c_void_p
_i32, _i64, _f64, _sz = ctypes.c_int32, ctypes.c_int64, ctypes.c_double, ctypes.c_size_t

_lib.ripple_alloc_budgets.argtypes = [ctypes.POINTER(_f64), _i32, _f64, _f64, _i64,
                                      ctypes.POINTER(_i64)]
_lib.ripple_alloc_budgets.restype = _i32
_lib.ripple_keep_count.argtypes = [_i64, _i32, _i32]
_lib.ripple_keep_count.restype = _i32
_lib.ripple_compress_workspace_bytes.argtypes = [ctypes.POINTER(LayerDesc), ctypes.POINTER(_sz)]
_lib.ripple_compress_workspace_bytes.restype = _i32
_lib.ripple_compress_layer.argtypes = [ctypes.POINTER(LayerDesc), _i64, _p, _p, _p, _p, _p, _i32,
                                       _p, _p, ctypes.POINTER(_i32), _p, _sz, _p, _p]
_lib.ripple_compress_layer.restype = _i32
_lib.ripple_compress_layers_workspace_bytes.argtypes = [ctypes.POINTER(LayerDesc), _i32,
                                                        ctypes.POINTER(_sz)]
_lib.ripple_compress_layers_workspace_bytes.restype = _i32
_lib.ripple_compress_layers.argtypes = [ctypes.POINTER(LayerDesc), _i32, ctypes.POINTER(_i64),
                                        ctypes.POINTER(_p), ctypes.POINTER(_p), ctypes.POINTER(_p),
                                        ctypes.POINTER(_p), ctypes.POINTER(_p),
                                        ctypes.POINTER(_i32), ctypes.POINTER(_p),
                                        ctypes.POINTER(_i32), _p, _sz, _p, _p]
_lib.ripple_compress_layers.restype = _i32
_lib.ripple_compress_layers_attn_workspace_bytes.argtypes = [ctypes.POINTER(LayerDesc), _i32,
                                                             ctypes.POINTER(_sz)]
_lib.ripple_compress_layers_attn_workspace_bytes.restype = _i32
_lib.ripple_compress_layers_attn.argtypes = [ctypes.POINTER(LayerDesc), _i32,
                                             ctypes.POINTER(_i64), ctypes.POINTER(_p),
                                             ctypes.POINTER(_p), ctypes.POINTER(_p),
                                             ctypes.POINTER(_p), ctypes.POINTER(_p),
                                             ctypes.POINTER(_i32), ctypes.POINTER(_p),
                                             ctypes.POINTER(_i32), ctypes.POINTER(_p), _p, _sz,
                                             _p, _p]
_lib.ripple_compress_layers_attn.restype = _i32
_lib.ripple_select_layer.argtypes = [ctypes.POINTER(LayerDesc), _i64, _p, _p, _p, _p, _p, _i32, _p,
                                     ctypes.POINTER(_i32), _p, _sz, _p, _p]
_lib.ripple_select_layer.restype = _i32
_lib.ripple_decode_workspace_bytes.argtypes = [ctypes.POINTER(DecodeDesc), ctypes.POINTER(_i32),
                                               ctypes.POINTER(_sz)]
_lib.ripple_decode_workspace_bytes.restype = _i32
_lib.ripple_decode_attn.argtypes = [ctypes.POINTER(DecodeDesc), _p, _p, _p, ctypes.POINTER(_p),
                                    ctypes.POINTER(_p), ctypes.POINTER(_i32), _p, _p, _p, _sz, _p,
                                    _p]
_lib.ripple_decode_attn.restype = _i32
_lib.ripple_decode_attn_noalloc.argtypes = [ctypes.POINTER(DecodeDesc), _p, _p, _p,
                                            ctypes.POINTER(_p), ctypes.POINTER(_p),
                                            ctypes.POINTER(_i32), _p, _p, _p, _p]
_lib.ripple_decode_attn_noalloc.restype = _i32
_lib.ripple_perturb_values.argtypes = [ctypes.POINTER(CacheDesc), _p, _p, ctypes.c_float, _i32,
                                       _i32, _p, _p]
_lib.ripple_perturb_values.restype = _i32
_lib.ripple_window_kl_workspace_bytes.argtypes = [_i32, _i32, _i32, ctypes.POINTER(_sz)]
_lib.ripple_window_kl_workspace_bytes.restype = _i32
_lib.ripple_window_kl.argtypes = [_p, _p, _i32, _i32, _i32, _i32, _p, _p, _p, _sz, _p, _p]
_lib.ripple_window_kl.restype = _i32
_lib.ripple_sensitivity_profile.argtypes = [ctypes.POINTER(_f64), _i32, _i32,
                                            ctypes.POINTER(_f64)]
_lib.ripple_sensitivity_profile.restype = _i32
_lib.ripple_set_wait_limit_cycles.argtypes = [_i64]
_lib.ripple_set_wait_limit_cycles.restype = _i64
_lib.ripple_kernel_launches.argtypes = []
_lib.ripple_kernel_launches.restype = ctypes.c_uint64
_lib.ripple_status_string.argtypes = [_i32]
_lib.ripple_status_string.restype = ctypes.c_char_p


def status_string(status: int) -> str:
    return _lib.ripple_status_string(int(status)).decode()


def _check(status: int, where: str):
    if status != OK:
        raise RippleError(status, where)


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


def layer_desc(batch, n_q_heads, n_kv_heads, head_dim, seq_len, window, pool_kernel=7,
               pool="max", dtype=torch.bfloat16, scale=0.0) -> LayerDesc:
    return LayerDesc(batch, n_q_heads, n_kv_heads, head_dim, seq_len, window, pool_kernel,
                     _POOLS[pool], _DTYPES[dtype], scale)


def decode_desc(n_layers, batch, n_q_heads, n_kv_heads, head_dim, dtype=torch.bfloat16,
                scale=0.0) -> DecodeDesc:
    return DecodeDesc(n_layers, batch, n_q_heads, n_kv_heads, head_dim, _DTYPES[dtype], scale)


# ----------------------------------------------------------------- entry points


def ripple_alloc_budgets(sens, ratio: float, gamma: float, global_budget: int) -> list:
    """Per-layer budgets b_l (Eqs. 9-12 with Eq. 5), computed by the host C allocator."""
    n = len(sens)
    s = (_f64 * n)(*[float(x) for x in sens])
    out = (_i64 * n)()
    _check(_lib.ripple_alloc_budgets(s, n, float(ratio), float(gamma), int(global_budget), out),
           "ripple_alloc_budgets")
    return [int(x) for x in out]


def ripple_keep_count(budget: int, seq_len: int, window: int) -> int:
    n = _lib.ripple_keep_count(int(budget), int(seq_len), int(window))
    if n < 0:
        raise RippleError(EINVAL, "ripple_keep_count")
    return n


def ripple_compress_workspace_bytes(desc: LayerDesc) -> int:
    out = _sz()
    _check(_lib.ripple_compress_workspace_bytes(ctypes.byref(desc), ctypes.byref(out)),
           "ripple_compress_workspace_bytes")
    return out.value


def ripple_compress_layer(desc: LayerDesc, budget: int, q_win, k, v, k_out, v_out, idx_out,
                          workspace, scores_out=None, dev_status=None, stream=None) -> int:
    """Compress one layer; returns n, the tokens kept per (batch, kv head).

    k_out/v_out are [B][Hkv][cap][d]; idx_out holds at least B*Hkv*n int32.
    """
    cap = k_out.shape[-2]
    n = _i32()
    _check(_lib.ripple_compress_layer(ctypes.byref(desc), int(budget), _ptr(q_win), _ptr(k),
                                      _ptr(v), _ptr(k_out), _ptr(v_out), cap, _ptr(idx_out),
                                      _ptr(scores_out), ctypes.byref(n), _ptr(workspace),
                                      workspace.numel() * workspace.element_size(),
                                      _ptr(dev_status), _stream(stream)),
           "ripple_compress_layer")
    return n.value


def ripple_compress_layers_workspace_bytes(desc: LayerDesc, n_layers: int) -> int:
    out = _sz()
    _check(_lib.ripple_compress_layers_workspace_bytes(ctypes.byref(desc), int(n_layers),
                                                       ctypes.byref(out)),
           "ripple_compress_layers_workspace_bytes")
    return out.value


class CompressTables:
    """Host arrays of per-layer device pointers for ripple_compress_layers,
    built once for a set of layer tensors (lists with one entry per layer)."""

    def __init__(self, q_win, k, v, k_out, v_out, idx_out):
        L = len(k)
        self.n_layers = L
        arr = lambda ts: (_p * L)(*[_ptr(x) for x in ts])
        self.q, self.k, self.v = arr(q_win), arr(k), arr(v)
        self.k_out, self.v_out, self.idx = arr(k_out), arr(v_out), arr(idx_out)
        self.caps = (_i32 * L)(*[int(x.shape[-2]) for x in k_out])
        self._keep = (list(q_win), list(k), list(v), list(k_out), list(v_out), list(idx_out))


def ripple_compress_layers(desc: LayerDesc, budgets, tables: CompressTables, workspace,
                           dev_status=None, stream=None) -> list:
    """Compress tables.n_layers layers of one shape in one call; returns n_l per layer."""
    L = tables.n_layers
    b = (_i64 * L)(*[int(x) for x in budgets])
    n = (_i32 * L)()
    _check(_lib.ripple_compress_layers(ctypes.byref(desc), L, b, tables.q, tables.k, tables.v,
                                       tables.k_out, tables.v_out, tables.caps, tables.idx, n,
                                       _ptr(workspace),
                                       workspace.numel() * workspace.element_size(),
                                       _ptr(dev_status), _stream(stream)),
           "ripple_compress_layers")
    return [int(x) for x in n]


def ripple_compress_layers_attn_workspace_bytes(desc: LayerDesc, n_layers: int) -> int:
    out = _sz()
    _check(_lib.ripple_compress_layers_attn_workspace_bytes(ctypes.byref(desc), int(n_layers),
                                                            ctypes.byref(out)),
           "ripple_compress_layers_attn_workspace_bytes")
    return out.value


def ripple_compress_layers_attn(desc: LayerDesc, budgets, tables: CompressTables, o_win,
                                workspace, dev_status=None, stream=None) -> list:
    """ripple_compress_layers that also writes each layer's window-row attention
    output into o_win[l] (fp32 [B][Hq][w][d]); returns n_l per layer."""
    L = tables.n_layers
    if len(o_win) != L:
        raise ValueError("one o_win tensor per layer")
    b = (_i64 * L)(*[int(x) for x in budgets])
    n = (_i32 * L)()
    o = (_p * L)(*[_ptr(x) for x in o_win])
    _check(_lib.ripple_compress_layers_attn(ctypes.byref(desc), L, b, tables.q, tables.k,
                                            tables.v, tables.k_out, tables.v_out, tables.caps,
                                            tables.idx, n, o, _ptr(workspace),
                                            workspace.numel() * workspace.element_size(),
                                            _ptr(dev_status), _stream(stream)),
           "ripple_compress_layers_attn")
    return [int(x) for x in n]


def ripple_select_layer(desc: LayerDesc, budget: int, votes, k, v, k_out, v_out, idx_out,
                        workspace, dev_status=None, stream=None) -> int:
    """Pool, select and gather one layer from given fp32 votes [B][Hkv][P]; returns n."""
    cap = k_out.shape[-2]
    n = _i32()
    _check(_lib.ripple_select_layer(ctypes.byref(desc), int(budget), _ptr(votes), _ptr(k), _ptr(v),
                                    _ptr(k_out), _ptr(v_out), cap, _ptr(idx_out), ctypes.byref(n),
                                    _ptr(workspace), workspace.numel() * workspace.element_size(),
                                    _ptr(dev_status), _stream(stream)),
           "ripple_select_layer")
    return n.value


def ripple_decode_workspace_bytes(desc: DecodeDesc, caps) -> int:
    c = (_i32 * len(caps))(*[int(x) for x in caps])
    out = _sz()
    _check(_lib.ripple_decode_workspace_bytes(ctypes.byref(desc), c, ctypes.byref(out)),
           "ripple_decode_workspace_bytes")
    return out.value


class DecodeTables:
    """Host arrays (cache pointers, capacities) of ripple_decode_attn, built once."""

    def __init__(self, k_caches, v_caches):
        L = len(k_caches)
        self.k = (_p * L)(*[_ptr(t) for t in k_caches])
        self.v = (_p * L)(*[_ptr(t) for t in v_caches])
        self.caps = (_i32 * L)(*[int(t.shape[-2]) for t in k_caches])
        self._keep = (list(k_caches), list(v_caches))


def ripple_decode_attn(desc: DecodeDesc, q, k_new, v_new, tables: DecodeTables, lens, out,
                       workspace, dev_status=None, stream=None):
    """One decode step over desc.n_layers layers: append, attend, advance lens."""
    _check(_lib.ripple_decode_attn(ctypes.byref(desc), _ptr(q), _ptr(k_new), _ptr(v_new),
                                   tables.k, tables.v, tables.caps, _ptr(lens), _ptr(out),
                                   _ptr(workspace), workspace.numel() * workspace.element_size(),
                                   _ptr(dev_status), _stream(stream)),
           "ripple_decode_attn")


NOALLOC_SCRATCH_BYTES = 8 << 20


def ripple_decode_attn_noalloc(desc: DecodeDesc, q, k_new, v_new, tables: DecodeTables, lens,
                               out, dev_status=None, stream=None):
    """ripple_decode_attn without a workspace argument, for callers that cannot
    allocate device memory (for instance a plugin whose host owns every device
    buffer and only passes tensors in and out). The split-K partials live in
    the library's own fixed device array of NOALLOC_SCRATCH_BYTES; steps that
    need more raise RippleError(EWORKSPACE). Calls overlapping on the GPU race
    on that array."""
    _check(_lib.ripple_decode_attn_noalloc(ctypes.byref(desc), _ptr(q), _ptr(k_new), _ptr(v_new),
                                           tables.k, tables.v, tables.caps, _ptr(lens),
                                           _ptr(out), _ptr(dev_status), _stream(stream)),
           "ripple_decode_attn_noalloc")


# ----------------------------------------------------- sensitivity profiling


def ripple_perturb_values(v, eps, alpha: float, pos_begin: int, pos_end: int, v_out=None,
                          stream=None):
    """Eq. 6 on one layer's Value cache v [B][Hkv][T][d]: rows in
    [pos_begin, pos_end) get v + alpha * ||v||_2 * eps (eps fp32
    [B][Hkv][pos_end - pos_begin][d]). In place when v_out is None, else into
    v_out (the other rows copied)."""
    B, H, T, d = v.shape
    desc = CacheDesc(B, H, T, d, _DTYPES[v.dtype])
    out = v if v_out is None else v_out
    _check(_lib.ripple_perturb_values(ctypes.byref(desc), _ptr(v), _ptr(eps), float(alpha),
                                      int(pos_begin), int(pos_end), _ptr(out), _stream(stream)),
           "ripple_perturb_values")


def ripple_window_kl_workspace_bytes(n_sets: int, n_pos: int, vocab: int) -> int:
    out = _sz()
    _check(_lib.ripple_window_kl_workspace_bytes(int(n_sets), int(n_pos), int(vocab),
                                                 ctypes.byref(out)),
           "ripple_window_kl_workspace_bytes")
    return out.value


def ripple_window_kl(p_logits, q_logits, workspace, d_out, kl_out=None, dev_status=None,
                     stream=None):
    """Eq. 7 for every set s: d_out[s] = mean over window positions t of
    KL(softmax(p_logits[t]) || softmax(q_logits[s][t])); p_logits [n_pos][V],
    q_logits [n_sets][n_pos][V] (same dtype), kl_out [n_sets][n_pos] or None."""
    n_sets, n_pos, vocab = q_logits.shape
    if tuple(p_logits.shape) != (n_pos, vocab) or p_logits.dtype != q_logits.dtype:
        raise ValueError("p_logits must be [n_pos][vocab] with q_logits' dtype")
    _check(_lib.ripple_window_kl(_ptr(p_logits), _ptr(q_logits), n_sets, n_pos, vocab,
                                 _DTYPES[q_logits.dtype], _ptr(kl_out), _ptr(d_out),
                                 _ptr(workspace), workspace.numel() * workspace.element_size(),
                                 _ptr(dev_status), _stream(stream)),
           "ripple_window_kl")


def ripple_sensitivity_profile(d) -> list:
    """Eq. 8 (host C): s_l = mean over the calibration examples of d[i][l]."""
    n, L = len(d), len(d[0]) if len(d) else 0
    flat = (_f64 * (n * L))(*[float(x) for row in d for x in row])
    out = (_f64 * max(L, 1))()
    _check(_lib.ripple_sensitivity_profile(flat, n, L, out), "ripple_sensitivity_profile")
    return [float(out[i]) for i in range(L)]


def ripple_kernel_launches() -> int:
    """Kernels the library has launched in this process."""
    return int(_lib.ripple_kernel_launches())


def ripple_set_wait_limit_cycles(cycles: int) -> int:
    """Bound of the in-kernel waits of later launches (SM cycles; <= 0 restores
    the default of about two seconds); returns the previous bound."""
    return int(_lib.ripple_set_wait_limit_cycles(int(cycles)))
