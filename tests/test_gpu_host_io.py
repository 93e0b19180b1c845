"""Per-step activations in page-locked host memory: the kernels read q, k, v
and write out in place over the host link, and every result is the same,
bit for bit, as with device tensors (the same kernels run; only the
addresses differ).  Pageable host memory is refused before any launch.
Every call goes through the C ABI (liboptr.so)."""
import ctypes

import pytest
import torch

from paper_2608_02691_gb300 import optr, synth

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02691_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def _pinned(t):
    return t.cpu().contiguous().pin_memory()


def _filled_case(name, scale, group=32, **kw):
    c = synth.build_case(synth.workload(name, 0, scale), 0)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"], group=group, **kw)
    pool = optr.new_pool(p, c["num_pages"], device=DEV)
    bt = c["block_table"].to(DEV)
    optr.optr_kv_append(p, c["k_ctx"].to(DEV), c["v_ctx"].to(DEV),
                        c["cu_ctx"].to(DEV), c["pos0_ctx"].to(DEV), bt, pool)
    return c, p, pool, bt


@pytest.mark.parametrize("variant", [optr.OPTR_VARIANT_CUDA_CORE, optr.OPTR_VARIANT_TENSOR])
@pytest.mark.parametrize("group", [32, 128])
def test_step_with_host_activations_is_bit_identical(variant, group):
    c, p, pool, bt = _filled_case("decode8k", 1 / 16, group=group, decode_variant=variant)
    pool_h = pool.clone()
    seq = c["seq_lens"].to(DEV)
    cu, pos0 = c["cu_new"].to(DEV), c["pos0_new"].to(DEV)
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device=DEV)
    out_d = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device=DEV)
    out_h = torch.full((c["B"], c["h_q"], 128), 7.0, dtype=torch.float32).pin_memory()
    optr.optr_decode_step(p, c["q"].to(DEV), c["k_new"].to(DEV), c["v_new"].to(DEV),
                          cu, pos0, bt, seq, pool, out_d, ws)
    optr.optr_decode_step(p, _pinned(c["q"]), _pinned(c["k_new"]), _pinned(c["v_new"]),
                          cu, pos0, bt, seq, pool_h, out_h, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    assert torch.equal(pool, pool_h)
    assert torch.equal(out_d.cpu(), out_h)


def test_decode_with_host_query_and_output_is_bit_identical():
    c, p, pool, bt = _filled_case("ragged", 1 / 32)
    seq = c["seq_lens_ctx"].to(DEV)  # decode over the context written above
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device=DEV)
    out_d = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device=DEV)
    out_h = torch.zeros(c["B"], c["h_q"], 128, dtype=torch.float32).pin_memory()
    optr.optr_decode_attention(p, c["q"].to(DEV), bt, seq, pool, out_d, ws)
    optr.optr_decode_attention(p, _pinned(c["q"]), bt, seq, pool, out_h, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    assert torch.equal(out_d.cpu(), out_h)


@pytest.mark.parametrize("scale", [1 / 512, 1 / 64])  # 256 and 2048 new tokens
def test_append_from_host_inputs_matches_the_cuda_core_write(scale):
    """A cache write from pinned host k, v runs on the CUDA-core kernel at
    any size (no TMA on host memory) and writes the same bytes as that
    kernel does from device inputs."""
    c = synth.build_case(synth.workload("prefill", 0, scale), 0)
    pools = []
    for host in (False, True):
        p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                    append_variant=optr.OPTR_VARIANT_CUDA_CORE if not host
                                    else optr.OPTR_VARIANT_TENSOR)
        pool = optr.new_pool(p, c["num_pages"], device=DEV)
        k = _pinned(c["k_new"]) if host else c["k_new"].to(DEV)
        v = _pinned(c["v_new"]) if host else c["v_new"].to(DEV)
        optr.optr_kv_append(p, k, v, c["cu_new"].to(DEV), c["pos0_new"].to(DEV),
                            c["block_table"].to(DEV), pool)
        torch.cuda.synchronize()
        assert optr.optr_device_error(p) == 0
        pools.append(pool)
    assert c["k_new"].shape[0] >= 256
    assert torch.equal(pools[0], pools[1])


def test_host_step_replays_from_a_cuda_graph():
    c, p, pool, bt = _filled_case("decode8k", 1 / 16)
    pool0 = pool.clone()
    seq = c["seq_lens"].to(DEV)
    cu, pos0 = c["cu_new"].to(DEV), c["pos0_new"].to(DEV)
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device=DEV)
    qh, kh, vh = _pinned(c["q"]), _pinned(c["k_new"]), _pinned(c["v_new"])
    out_h = torch.zeros(c["B"], c["h_q"], 128, dtype=torch.float32).pin_memory()
    ref = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device=DEV)
    optr.optr_decode_step(p, c["q"].to(DEV), c["k_new"].to(DEV), c["v_new"].to(DEV),
                          cu, pos0, bt, seq, pool0, ref, ws)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            optr.optr_decode_step(p, qh, kh, vh, cu, pos0, bt, seq, pool, out_h, ws,
                                  stream=s)
    for _ in range(2):
        out_h.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(out_h, ref.cpu())
    assert torch.equal(pool, pool0)
    assert optr.optr_device_error(p) == 0


def test_pageable_host_memory_is_refused():
    """Through the C ABI directly (the binding refuses unpinned tensors
    itself): a pageable q or out gives OPTR_ERR_INVALID_ARG, nothing runs."""
    c, p, pool, bt = _filled_case("tiny", 1.0)
    seq = c["seq_lens"].to(DEV)
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device=DEV)
    q_pageable = c["q"].cpu().contiguous()
    out_d = torch.full((c["B"], c["h_q"], 128), 3.0, dtype=torch.float32, device=DEV)
    out_pageable = torch.zeros(c["B"], c["h_q"], 128, dtype=torch.float32)
    assert not q_pageable.is_pinned()
    lib = optr.lib()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    B, max_pages = bt.shape
    for q, out in ((q_pageable, out_d), (c["q"].to(DEV), out_pageable)):
        st = lib.optr_decode_attention(
            p.handle, ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(bt.data_ptr()),
            ctypes.c_void_p(seq.data_ptr()), B, max_pages, ctypes.c_void_p(pool.data_ptr()),
            pool.shape[0], ctypes.c_void_p(out.data_ptr()), ctypes.c_void_p(ws.data_ptr()),
            ws.numel(), stream)
        assert st == -1  # OPTR_ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert torch.all(out_d == 3.0)
    with pytest.raises(ValueError):
        optr.optr_decode_attention(p, q_pageable, bt, seq, pool, out_d, ws)


def test_windowed_step_with_host_activations_is_bit_identical():
    """The paper's default configuration (G = 128, clips 0.96 / 0.92, BF16
    sink 64 / recent 256 windows): a step from pinned host buffers writes
    the same pool and window bytes and returns the same output."""
    c = synth.build_case(synth.workload("decode8k", 0, 1 / 16), 0)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"], group=128,
                                clip_k=0.96, clip_v=0.92, sink=64, recent=256)
    bt = c["block_table"].to(DEV)
    slot = torch.arange(c["B"], dtype=torch.int32, device=DEV)
    pool = optr.new_pool(p, c["num_pages"], device=DEV)
    win = optr.new_windows(p, c["B"], device=DEV)
    optr.optr_kv_append_win(p, c["k_ctx"].to(DEV), c["v_ctx"].to(DEV), c["cu_ctx"].to(DEV),
                            c["pos0_ctx"].to(DEV), bt, pool, win, slot)
    pool_h, win_h = pool.clone(), win.clone()
    seq = c["seq_lens"].to(DEV)
    cu, pos0 = c["cu_new"].to(DEV), c["pos0_new"].to(DEV)
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device=DEV)
    out_d = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device=DEV)
    out_h = torch.zeros(c["B"], c["h_q"], 128, dtype=torch.float32).pin_memory()
    optr.optr_decode_step_win(p, c["q"].to(DEV), c["k_new"].to(DEV), c["v_new"].to(DEV),
                              cu, pos0, bt, seq, pool, win, slot, out_d, ws)
    optr.optr_decode_step_win(p, _pinned(c["q"]), _pinned(c["k_new"]), _pinned(c["v_new"]),
                              cu, pos0, bt, seq, pool_h, win_h, slot, out_h, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    assert torch.equal(pool, pool_h)
    assert torch.equal(win, win_h)
    assert torch.equal(out_d.cpu(), out_h)


def test_windowed_prefill_from_host_inputs():
    """A windowed cache write of a whole context (more than 256 tokens:
    the CUDA-core kernel, then the window-copy kernel) from pinned host k, v
    writes the same pool and window bytes as from device inputs."""
    c = synth.build_case(synth.workload("decode8k", 0, 1 / 16), 0)
    out = []
    for host in (False, True):
        p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                    append_variant=optr.OPTR_VARIANT_CUDA_CORE,
                                    sink=64, recent=256)
        pool = optr.new_pool(p, c["num_pages"], device=DEV)
        win = optr.new_windows(p, c["B"], device=DEV)
        slot = torch.arange(c["B"], dtype=torch.int32, device=DEV)
        k = _pinned(c["k_ctx"]) if host else c["k_ctx"].to(DEV)
        v = _pinned(c["v_ctx"]) if host else c["v_ctx"].to(DEV)
        optr.optr_kv_append_win(p, k, v, c["cu_ctx"].to(DEV), c["pos0_ctx"].to(DEV),
                                c["block_table"].to(DEV), pool, win, slot)
        torch.cuda.synchronize()
        assert optr.optr_device_error(p) == 0
        out.append((pool, win))
    assert c["k_ctx"].shape[0] > 256
    assert torch.equal(out[0][0], out[1][0])
    assert torch.equal(out[0][1], out[1][1])
