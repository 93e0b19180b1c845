"""CPU-only checks of the C ABI boundary and the host-side split-K logic.

No test here launches a kernel: the library is loaded, its exported symbols
are compared with include/optr.h, and argument errors that the host rejects
before touching CUDA are exercised.
"""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "optr.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_02691_gb300 import build, optr
    build.build()
    return optr.lib()


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(optr_[a-z_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("optr_params_create", "optr_params_destroy", "optr_kv_append",
              "optr_decode_workspace_size", "optr_decode_attention",
              "optr_device_error", "optr_strerror", "optr_page_bytes"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_strerror_covers_every_status(lib):
    from paper_2608_02691_gb300 import optr
    for s in range(-5, 1):
        assert optr.optr_strerror(s) and "unknown" not in optr.optr_strerror(s)
    assert "unknown" in optr.optr_strerror(-99)


def test_host_argument_errors_launch_nothing(lib):
    from paper_2608_02691_gb300 import optr
    cfg = optr.optr_config(32, 8, 128, 32, 16, 1.0, 1.0, 0, 0)
    h = ctypes.c_void_p()
    f = (ctypes.c_float * 4)()
    # null matrices / handle
    assert lib.optr_params_create(ctypes.byref(cfg), None, f, f, ctypes.byref(h)) == -1
    assert lib.optr_params_create(None, f, f, f, ctypes.byref(h)) == -1
    # unsupported shapes: head_dim, group, page size, GQA ratio
    for bad in (dict(head_dim=64), dict(group=64), dict(page_size=8),
                dict(h_q=16)):
        c = optr.optr_config(32, 8, 128, 32, 16, 1.0, 1.0, 0, 0)
        for k, val in bad.items():
            setattr(c, k, val)
        assert lib.optr_params_create(ctypes.byref(c), f, f, f, ctypes.byref(h)) == -2
    c = optr.optr_config(32, 8, 128, 32, 16, 0.0, 1.0, 0, 0)
    assert lib.optr_params_create(ctypes.byref(c), f, f, f, ctypes.byref(h)) == -1
    # BF16 windows: sink a multiple of 16, both windows at most 1024
    for sink, recent, want in ((8, 0, -1), (-16, 0, -1), (0, -1, -1),
                               (1040, 0, -3), (0, 1025, -3)):
        c = optr.optr_config(32, 8, 128, 32, 16, 1.0, 1.0, 0, 0, sink, recent)
        assert lib.optr_params_create(ctypes.byref(c), f, f, f, ctypes.byref(h)) == want
    assert not h.value
    # operations on a null handle
    assert lib.optr_kv_append(None, None, None, 1, None, None, None, 1, 1,
                              None, 1, None) == -1
    assert lib.optr_decode_attention(None, None, None, None, 1, 1, None, 1,
                                     None, None, 0, None) == -1
    assert lib.optr_decode_step(None, None, None, None, 0, None, None, None,
                                None, 1, 1, None, 1, None, None, 0, None) == -1
    assert lib.optr_decode_attention_noalloc(None, None, None, None, 1, 1,
                                             None, 1, None, None) == -1
    assert lib.optr_decode_workspace_size(None, 1, 1) == 0
    assert lib.optr_page_bytes(None) == 0
    # the BF16-window entry points
    assert lib.optr_window_bytes(None, 4) == 0
    assert lib.optr_kv_append_win(None, None, None, 1, None, None, None, 1, 1,
                                  None, 1, None, None, 0, None) == -1
    assert lib.optr_decode_attention_win(None, None, None, None, 1, 1, None, 1,
                                         None, None, 0, None, None, 0,
                                         None) == -1
    assert lib.optr_decode_step_win(None, None, None, None, 0, None, None, None,
                                    None, 1, 1, None, 1, None, None, 0, None,
                                    None, 0, None) == -1
    flags = ctypes.c_uint32()
    assert lib.optr_device_error(None, ctypes.byref(flags)) == -1


# ---------------------------------------------------------- split-K plan

def test_window_unit_partition_gives_each_window_warp_work():
    """BF16-window units: Ww = min(window warps, units), contiguous ranges;
    every window warp owns at least one unit, and the warps owning a
    sequence's non-empty units form a gap-free run whose closed-form ends
    (the combine's) are the first and last owner."""
    import random
    rng = random.Random(3)
    for _ in range(300):
        B, h_kv, Uw = rng.randint(1, 40), rng.choice([1, 8]), rng.choice([1, 4, 20])
        U = B * h_kv * Uw
        Ww = min(rng.choice([7, 64, 608]), U)
        owner = {}
        for w in range(Ww):
            u0, u1 = w * U // Ww, (w + 1) * U // Ww
            assert u1 > u0
            for u in range(u0, u1):
                owner[u] = w
        for bh in range(B * h_kv):
            nwu = rng.randint(0, Uw)
            if nwu == 0:
                continue
            ws = [owner[bh * Uw + j] for j in range(nwu)]
            assert ws == sorted(ws) and set(ws) == set(range(ws[0], ws[-1] + 1))
            assert _warp_of(bh * Uw, U, Ww) == ws[0]
            assert _warp_of(bh * Uw + nwu - 1, U, Ww) == ws[-1]


def _ranges(F, W):
    return [(w * F // W, (w + 1) * F // W) for w in range(W)]


def _warp_of(f, F, W):
    return min(W - 1, ((f + 1) * W - 1) // F)


@pytest.mark.parametrize("F,W", [(1, 7), (5, 7), (7, 7), (8, 7), (1000, 7),
                                 (2431, 2432), (4096 * 8, 2432), (999983, 2432)])
def test_warp_partition_owner_formula(F, W):
    """Each flat page index belongs to exactly one warp range, and the
    closed-form owner used by the combine kernel names that warp."""
    rs = _ranges(F, W)
    assert rs[0][0] == 0 and rs[-1][1] == F
    assert all(a[1] == b[0] for a, b in zip(rs, rs[1:]))
    step = max(1, F // 5000)
    for f in list(range(0, F, step)) + [F - 1]:
        w = _warp_of(f, F, W)
        assert rs[w][0] <= f < rs[w][1]


def test_partial_slots_are_unique():
    """Slot w + idx(b, h) is unique over all (warp, segment) pairs: walk the
    same segmentation the partial kernel performs."""
    import random
    rnd = random.Random(0)
    for trial in range(30):
        B = rnd.randint(1, 40)
        H = rnd.choice([1, 2, 8])
        np_ = [rnd.choice([0, 0, 1, 2, 3, 17, 64]) for _ in range(B)]
        pref = [0]
        nz = [0]
        for n in np_:
            pref.append(pref[-1] + n)
            nz.append(nz[-1] + (n > 0))
        F = pref[-1] * H
        if F == 0:
            continue
        W = rnd.choice([1, 3, 16, 200])
        seen = set()
        count = {}
        for w, (f, f1) in enumerate(_ranges(F, W)):
            while f < f1:
                b = max(i for i in range(B) if pref[i] * H <= f)
                n = pref[b + 1] - pref[b]
                assert n > 0
                base = pref[b] * H
                h = (f - base) // n
                end = min(f1, base + (h + 1) * n)
                slot = w + nz[b] * H + h
                assert slot not in seen and slot < W + B * H
                seen.add(slot)
                count[(b, h)] = count.get((b, h), 0) + 1
                f = end
        for (b, h), c in count.items():
            n = pref[b + 1] - pref[b]
            fs = pref[b] * H + h * n
            owners = [w for w in range(_warp_of(fs, F, W), _warp_of(fs + n - 1, F, W) + 1)
                      if w * F // W != (w + 1) * F // W]  # skip empty ranges
            assert len(owners) == c
