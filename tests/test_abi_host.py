"""The C-ABI library without a GPU: it loads, exports every declared symbol,
its host allocator matches the oracle bit for bit, and host-side argument
validation rejects bad calls before any CUDA work."""
import ctypes
import math
import os
import random
import re

import pytest

from oracle import ripple_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    names = []
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names += re.findall(r"^\s*[A-Za-z_][\w\s\*]*?\b(ripple_\w+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = _declared_functions()
    for n in ("ripple_alloc_budgets", "ripple_compress_layer", "ripple_decode_attn"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    raw = ctypes.CDLL(lib.LIB_PATH)
    for name in _declared_functions():
        assert hasattr(raw, name), name


def _cases():
    rnd = random.Random(2024)
    out = []
    for _ in range(300):
        L = rnd.choice([1, 2, 3, 4, 5, 8, 31, 32, 80, 128])
        kind = rnd.random()
        if kind < 0.1:
            s = [0.25] * L
        elif kind < 0.2:
            s = [float(rnd.randint(0, 3)) for _ in range(L)]
        else:
            s = [rnd.lognormvariate(-4.0, 1.2) for _ in range(L)]
        r = rnd.choice([1.0, 1.25, 1.5, 1.75, 2.0, 4.0, 8.0, 32.0])
        gamma = rnd.choice([math.inf, 0.0, -1.0, 1.0, 1.5, 2.0, 4.0])
        B = rnd.choice([0, 1, 7, L, 3 * L + 1, 128 * L, 512 * L, 1024 * L + 13, 2048 * L])
        out.append((s, r, gamma, B))
    return out


def test_host_allocator_bit_exact_vs_oracle(lib):
    for s, r, gamma, B in _cases():
        assert lib.ripple_alloc_budgets(s, r, gamma, B) == O.alloc_budgets(s, r, gamma, B)


def test_host_allocator_worked_example(lib):
    assert lib.ripple_alloc_budgets([0.2, 1.0, 0.6, 0.1], 4.0, math.inf, 512) == [72, 246, 133, 61]


@pytest.mark.parametrize("args", [
    ([], 4.0, math.inf, 10),
    ([0.1, 0.2], 0.5, math.inf, 10),
    ([0.1, 0.2], math.inf, math.inf, 10),
    ([0.1, 0.2], math.nan, math.inf, 10),
    ([0.1, 0.2], 4.0, 0.5, 10),
    ([0.1, 0.2], 4.0, math.nan, 10),
    ([0.1, math.nan], 4.0, math.inf, 10),
    ([0.1, math.inf], 4.0, math.inf, 10),
    ([0.1, 0.2], 4.0, math.inf, -1),
])
def test_host_allocator_rejects_bad_arguments(lib, args):
    with pytest.raises(lib.RippleError) as e:
        lib.ripple_alloc_budgets(*args)
    assert e.value.status == lib.EINVAL


def test_keep_count_matches_oracle(lib):
    for b, T, w in [(100, 512, 32), (10, 512, 32), (5000, 512, 32), (0, 16, 16), (33, 33, 1)]:
        assert lib.ripple_keep_count(b, T, w) == O.keep_count(b, T, w)
    with pytest.raises(lib.RippleError):
        lib.ripple_keep_count(5, 10, 11)


def test_workspace_query_and_validation(lib):
    d = lib.layer_desc(4, 32, 8, 128, 32768, 32)
    assert lib.ripple_compress_workspace_bytes(d) > 4 * 8 * 32736 * 4
    bad = [lib.layer_desc(1, 6, 4, 128, 100, 8),   # Hq not a multiple of Hkv
           lib.layer_desc(1, 4, 2, 96, 100, 8),    # unsupported head_dim
           lib.layer_desc(1, 4, 2, 64, 100, 101),  # window > T
           lib.layer_desc(1, 4, 2, 64, 100, 8, pool_kernel=4),
           lib.layer_desc(1, 64, 1, 64, 100, 8)]   # G * w > 256
    for d in bad:
        with pytest.raises(lib.RippleError):
            lib.ripple_compress_workspace_bytes(d)


def test_entry_points_reject_before_any_cuda_work(lib):
    # NULL pointers / bad shapes are refused on the host; nothing is launched.
    raw = lib._lib
    d = lib.layer_desc(1, 4, 2, 64, 512, 32, dtype=__import__("torch").float32)
    n = ctypes.c_int32(-7)
    st = raw.ripple_compress_layer(ctypes.byref(d), 100, None, None, None, None, None, 128, None,
                                   None, ctypes.byref(n), None, 0, None, None)
    assert st == lib.EINVAL and n.value == -7
    dd = lib.decode_desc(2, 1, 4, 2, 64)
    st = raw.ripple_decode_attn(ctypes.byref(dd), None, None, None, None, None, None, None, None,
                                None, 0, None, None)
    assert st == lib.EINVAL
    assert lib.status_string(lib.EFULL) == "cache full"


def test_compress_layers_host_validation(lib):
    d = lib.layer_desc(4, 32, 8, 128, 32768, 32)
    one = lib.ripple_compress_workspace_bytes(d)
    four = lib.ripple_compress_layers_workspace_bytes(d, 4)
    assert four >= 4 * 4 * 8 * 32736 * 4 and four > one
    for bad in (0, -1, lib.COMPRESS_MAX_LAYERS + 1):
        with pytest.raises(lib.RippleError):
            lib.ripple_compress_layers_workspace_bytes(d, bad)
    raw = ctypes.CDLL(lib.LIB_PATH)
    n = (ctypes.c_int32 * 2)()
    st = raw.ripple_compress_layers(ctypes.byref(d), 2, None, None, None, None, None, None,
                                    None, None, n, None, 0, None, None)
    assert st == lib.EINVAL


def test_sensitivity_profile_bit_exact_vs_oracle(lib):
    rnd = random.Random(11)
    for _ in range(50):
        n, L = rnd.randint(1, 9), rnd.choice([1, 4, 32, 80])
        d = [[rnd.lognormvariate(-5.0, 1.5) for _ in range(L)] for _ in range(n)]
        assert lib.ripple_sensitivity_profile(d) == [float(x) for x in O.sensitivity_profile(d)]
    raw = lib._lib
    out = (ctypes.c_double * 2)()
    bad = (ctypes.c_double * 2)(1.0, math.nan)
    assert raw.ripple_sensitivity_profile(bad, 1, 2, out) == lib.EINVAL
    assert raw.ripple_sensitivity_profile(bad, 0, 2, out) == lib.EINVAL
    assert raw.ripple_sensitivity_profile(None, 1, 2, out) == lib.EINVAL


def test_profiling_entry_points_reject_before_any_cuda_work(lib):
    raw = lib._lib
    fake = 1 << 20  # aligned, never dereferenced: every call below fails validation first
    d = lib.CacheDesc(1, 2, 64, 128, lib.BF16)
    for args in [(fake, fake, 0.1, -1, 10, fake), (fake, fake, 0.1, 10, 65, fake),
                 (fake, fake, 0.1, 20, 10, fake), (fake, fake, -0.5, 0, 10, fake),
                 (fake, fake, math.inf, 0, 10, fake), (fake, None, 0.1, 0, 10, fake),
                 (fake + 8, fake, 0.1, 0, 10, fake), (None, fake, 0.1, 0, 10, fake)]:
        assert raw.ripple_perturb_values(ctypes.byref(d), *args, None) == lib.EINVAL, args
    for bad in (lib.CacheDesc(1, 2, 64, 96, lib.BF16), lib.CacheDesc(0, 2, 64, 128, lib.BF16),
                lib.CacheDesc(1, 2, 64, 128, 7)):
        assert raw.ripple_perturb_values(ctypes.byref(bad), fake, fake, 0.1, 0, 10, fake,
                                         None) == lib.EINVAL
    n = lib.ripple_window_kl_workspace_bytes(32, 32, 128256)
    assert n >= 32 * 32 * 16 * 20 and n % 256 == 0
    for args in [(0, 4, 64), (2, 0, 64), (2, 4, 12), (2, 4, 0)]:
        with pytest.raises(lib.RippleError):
            lib.ripple_window_kl_workspace_bytes(*args)
    kl = raw.ripple_window_kl
    assert kl(fake, fake, 2, 4, 64, lib.F32, None, fake, fake, 0, None, None) == lib.EWORKSPACE
    assert kl(fake, fake, 2, 4, 60, lib.F32, None, fake, fake, 1 << 30, None, None) == lib.EINVAL
    assert kl(fake, fake, 2, 4, 64, 5, None, fake, fake, 1 << 30, None, None) == lib.EINVAL
    assert kl(fake, None, 2, 4, 64, lib.F32, None, fake, fake, 1 << 30, None, None) == lib.EINVAL
    assert kl(fake, fake, 2, 4, 64, lib.F32, None, None, fake, 1 << 30, None, None) == lib.EINVAL
    assert kl(fake + 4, fake, 2, 4, 64, lib.F32, None, fake, fake, 1 << 30, None, None) == lib.EINVAL
    assert kl(fake, fake, 2, 4, 64, lib.F32, None, fake, fake + 16, 1 << 30, None, None) == lib.EINVAL


def test_compress_and_decode_argument_table(lib):
    # Every call below is invalid and must be refused on the host, outputs
    # untouched; none reaches a CUDA call (the fake pointers are never used).
    raw = lib._lib
    fake, mis = 1 << 20, (1 << 20) + 8
    d = lib.layer_desc(1, 4, 2, 128, 512, 32)
    need = lib.ripple_compress_workspace_bytes(d)
    base = dict(budget=100, q=fake, k=fake, v=fake, ko=fake, vo=fake, cap=128, idx=fake,
                scores=None, ws=fake, wsb=need)

    def compress(**over):
        a = dict(base, **over)
        n = ctypes.c_int32(-7)
        st = raw.ripple_compress_layer(ctypes.byref(d), a["budget"], a["q"], a["k"], a["v"],
                                       a["ko"], a["vo"], a["cap"], a["idx"], a["scores"],
                                       ctypes.byref(n), a["ws"], a["wsb"], None, None)
        assert n.value == -7, over
        return st

    for key in ("q", "k", "v", "ko", "vo", "idx", "ws"):
        assert compress(**{key: None}) == lib.EINVAL, key
        assert compress(**{key: mis}) == lib.EINVAL, key
    assert compress(scores=mis) == lib.EINVAL
    assert compress(ws=fake + 16) == lib.EINVAL  # workspace must be 256-byte aligned
    assert compress(budget=-1) == lib.EINVAL
    assert compress(cap=99) == lib.EINVAL        # n = 100 rows do not fit
    assert compress(wsb=need - 1) == lib.EWORKSPACE
    assert raw.ripple_select_layer(ctypes.byref(d), 100, None, fake, fake, fake, fake, 128, fake,
                                   ctypes.byref(ctypes.c_int32()), fake, need, None,
                                   None) == lib.EINVAL

    L = 2
    ptrs = lambda *xs: (ctypes.c_void_p * L)(*xs)
    caps = (ctypes.c_int32 * L)(16, 16)
    dd = lib.decode_desc(L, 1, 4, 2, 64)
    dneed = lib.ripple_decode_workspace_bytes(dd, [16, 16])

    def decode(desc=dd, q=fake, kc=None, vc=None, cp=caps, ws=fake, wsb=dneed):
        kc = kc if kc is not None else ptrs(fake, fake)
        vc = vc if vc is not None else ptrs(fake, fake)
        return raw.ripple_decode_attn(ctypes.byref(desc), q, fake, fake, kc, vc, cp, fake, fake,
                                      ws, wsb, None, None)

    for bad in (lib.decode_desc(L, 1, 6, 2, 64),          # G = 3
                lib.decode_desc(L, 1, 32, 2, 64),         # G = 16
                lib.decode_desc(0, 1, 4, 2, 64),
                lib.decode_desc(lib.MAX_LAYERS + 1, 1, 4, 2, 64),
                lib.decode_desc(L, 1, 4, 2, 80),
                lib.decode_desc(L, 1, 4, 2, 64, scale=-1.0)):
        assert decode(desc=bad) == lib.EINVAL
    assert decode(q=None) == lib.EINVAL
    assert decode(q=mis) == lib.EINVAL
    assert decode(kc=ptrs(fake, None)) == lib.EINVAL
    assert decode(vc=ptrs(mis, fake)) == lib.EINVAL
    assert decode(cp=(ctypes.c_int32 * L)(16, 0)) == lib.EINVAL
    assert decode(ws=None) == lib.EINVAL
    assert decode(ws=fake + 16) == lib.EINVAL
    assert decode(wsb=dneed - 1) == lib.EWORKSPACE
    assert raw.ripple_decode_attn_noalloc(ctypes.byref(lib.decode_desc(L, 1, 6, 2, 64)), fake,
                                          fake, fake, ptrs(fake, fake), ptrs(fake, fake), caps,
                                          fake, fake, None, None) == lib.EINVAL
