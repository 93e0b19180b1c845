"""The paper's default quantizer settings on the GPU (Sec. 5 and the
default-settings table: group size G = 128, clipping ratios 0.96 for keys
and 0.92 for values; with its 64 sink and 256 recent BF16 tokens), against
the oracle:

* cache write with G = 128 on every write path (single-token tiles of the
  decode step, the CUDA-core kernel for larger writes, which G = 128 writes
  use under every variant), codes and metadata as without;
* decode over oracle-written G = 128 pools, both decode variants;
* the whole paper-default configuration (G = 128, clips, windows) through
  the fused decode step.
"""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_02691_gb300 import optr, synth

import parity_helpers as ph

pytestmark = pytest.mark.gpu

VARIANTS = [optr.OPTR_VARIANT_CUDA_CORE, optr.OPTR_VARIANT_TENSOR]
CASES = [("tiny", 1.0), ("decode8k", 1 / 16), ("ragged", 1 / 32),
         ("prefill", 1 / 128)]
CK, CV = 0.96, 0.92


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02691_gb300 import build
    build.build()
    oracle.build()
    oracle.set_threads(max(1, min(16, __import__("os").cpu_count() or 1)))
    torch.cuda.set_device(0)


_cache = {}


def _case(name, scale):
    if (name, scale) not in _cache:
        c = synth.build_case(synth.workload(name, 0, scale), 0)
        _cache[(name, scale)] = (c, *ph.oracle_case(c, group=128, clip_k=CK, clip_v=CV))
    return _cache[(name, scale)]


@pytest.mark.parametrize("name,scale", CASES)
@pytest.mark.parametrize("avar", VARIANTS)
def test_group128_cache_write(name, scale, avar):
    c, pool_ref, u_ctx, u_new = _case(name, scale)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                clip_k=CK, clip_v=CV, append_variant=avar,
                                group=128)
    pool = optr.new_pool(p, c["num_pages"])
    bt = c["block_table"].cuda()
    for kk, vv, cu, pos0 in ((c["k_ctx"], c["v_ctx"], c["cu_ctx"], c["pos0_ctx"]),
                             (c["k_new"], c["v_new"], c["cu_new"], c["pos0_new"])):
        if kk.shape[0]:
            optr.optr_kv_append(p, kk.cuda(), vv.cuda(), cu.cuda(), pos0.cuda(),
                                bt, pool)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    pg = pool.cpu().numpy()
    for cu, pos0, u in ((c["cu_ctx"], c["pos0_ctx"], u_ctx),
                        (c["cu_new"], c["pos0_new"], u_new)):
        if u is None:
            continue
        pages, slots = ph.token_slots(cu, pos0, c["block_table"])
        st = ph.compare_append(pg, pool_ref, u, pages, slots)
    # the compact record: 1152 bytes per (page, KV head), and the bytes
    # between the metadata of the last slot and the next record untouched
    assert pg.shape[-1] == 1152
    written = np.zeros(pg.shape[:2], bool)
    for cu, pos0 in ((c["cu_ctx"], c["pos0_ctx"]), (c["cu_new"], c["pos0_new"])):
        pages, _ = ph.token_slots(cu, pos0, c["block_table"])
        written[pages] = True
    assert not pg[~written.any(axis=1)].any()  # pages no token maps to stay zero


@pytest.mark.parametrize("name,scale", CASES[:3])
@pytest.mark.parametrize("dvar", VARIANTS)
def test_group128_decode(name, scale, dvar):
    c, pool_ref, _, _ = _case(name, scale)
    got = ph.gpu_decode(c, pool_ref, variant=dvar)
    ref = ph.oracle_decode(c, pool_ref)
    ph.assert_decode_close(got, ref, f"{name} G=128")


@pytest.mark.parametrize("dvar", VARIANTS)
def test_paper_default_configuration_step(dvar):
    """G = 128, c_K = 0.96, c_V = 0.92, 64 sink and 256 recent BF16 tokens:
    context written, then the fused step (new token, decode)."""
    sink, recent = 64, 256
    c, pool_ref, u_ctx, u_new = _case("decode8k", 1 / 16)
    B = c["B"]
    slots = np.arange(B, dtype=np.int32)
    win_ref = oracle.new_windows(B, c["h_kv"], sink, recent)
    for kk, vv, cu, pos0 in ((c["k_ctx"], c["v_ctx"], c["cu_ctx"], c["pos0_ctx"]),
                             (c["k_new"], c["v_new"], c["cu_new"], c["pos0_new"])):
        oracle.window_write(synth.bf16_bits(kk), synth.bf16_bits(vv), cu.numpy(),
                            pos0.numpy(), win_ref, slots, sink, recent)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                clip_k=CK, clip_v=CV, decode_variant=dvar,
                                sink=sink, recent=recent, group=128)
    pool = optr.new_pool(p, c["num_pages"])
    win = optr.new_windows(p, B)
    ws_slot = torch.from_numpy(slots).cuda()
    bt = c["block_table"].cuda()
    optr.optr_kv_append_win(p, c["k_ctx"].cuda(), c["v_ctx"].cuda(),
                            c["cu_ctx"].cuda(), c["pos0_ctx"].cuda(), bt, pool,
                            win, ws_slot)
    out = torch.empty(B, c["h_q"], 128, dtype=torch.float32, device="cuda")
    ws = optr.new_workspace(p, B, bt.shape[1])
    optr.optr_decode_step_win(p, c["q"].cuda(), c["k_new"].cuda(),
                              c["v_new"].cuda(), c["cu_new"].cuda(),
                              c["pos0_new"].cuda(), bt, c["seq_lens"].cuda(),
                              pool, win, ws_slot, out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    assert np.array_equal(win.cpu().view(torch.int16).numpy().view(np.uint16), win_ref)
    pg = pool.cpu().numpy()
    diffs = []
    for cu, pos0, u in ((c["cu_ctx"], c["pos0_ctx"], u_ctx),
                        (c["cu_new"], c["pos0_new"], u_new)):
        pages, sl = ph.token_slots(cu, pos0, c["block_table"])
        st = ph.compare_append(pg, pool_ref, u, pages, sl)
        diffs.append((cu.numpy(), pos0.numpy(), st["flipped"]))
    ref = oracle.decode_attention(
        synth.bf16_bits(c["q"]), c["block_table"].numpy(), c["seq_lens"].numpy(),
        pool_ref, c["R_k"].numpy(), c["R_v"].numpy(), c["h_kv"], win=win_ref,
        win_slot=slots, sink=sink, recent=recent, mu=c["mu"].numpy())
    got = out.cpu().double().numpy()
    bound = ph.e2e_row_bounds(c, pool_ref, pg, diffs, win=win_ref,
                              win_slot=slots, sink=sink, recent=recent)
    strict, mean_bar = ph.assert_rows_within_bar(got, ref, bound, "paper defaults")
    print(f"paper defaults: strict rows {strict:.2f}, mean bar {mean_bar:.3f} x strict")


def test_compact_step_replays_from_a_cuda_graph():
    """The decode step on the compact G = 128 record (single-token write of
    one pair per slot, decode reading 1152-byte records) captured in a CUDA
    graph and replayed gives the bytes and output of direct calls."""
    c = synth.build_case(synth.workload("decode8k", 0, 1 / 32), 0)
    dev = "cuda"
    res = []
    for use_graph in (False, True):
        p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                    clip_k=CK, clip_v=CV, group=128)
        pool = optr.new_pool(p, c["num_pages"], device=dev)
        assert pool.shape[-1] == 1152
        bt = c["block_table"].to(dev)
        optr.optr_kv_append(p, c["k_ctx"].to(dev), c["v_ctx"].to(dev),
                            c["cu_ctx"].to(dev), c["pos0_ctx"].to(dev), bt, pool)
        args = [c["q"].to(dev), c["k_new"].to(dev), c["v_new"].to(dev),
                c["cu_new"].to(dev), c["pos0_new"].to(dev), bt,
                c["seq_lens"].to(dev)]
        out = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device=dev)
        ws = optr.new_workspace(p, c["B"], bt.shape[1], device=dev)
        torch.cuda.synchronize()
        if use_graph:
            s = torch.cuda.Stream()
            s.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(s):  # warm-up outside the capture
                optr.optr_decode_step(p, *args, pool, out, ws)
            torch.cuda.current_stream().wait_stream(s)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                optr.optr_decode_step(p, *args, pool, out, ws)
            out.zero_()
            g.replay()
        else:
            optr.optr_decode_step(p, *args, pool, out, ws)
            optr.optr_decode_step(p, *args, pool, out, ws)
        torch.cuda.synchronize()
        assert optr.optr_device_error(p) == 0
        res.append((pool.cpu(), out.cpu()))
    assert torch.equal(res[0][0], res[1][0])
    assert torch.equal(res[0][1], res[1][1])
