"""BF16 sink and recent windows on the GPU (Sec. 3.1: INT2 long history with
a small BF16 window; Sec. 4.1: window keys centered by the same mu; Sec. 5:
64 sink and 256 recent tokens), against the oracle:

* cache write: INT2 records as before, window store bit-exact (a copy);
* decode over the oracle-written pool and store, both decode variants,
  window shapes from the paper's (64, 256) to sink-only / recent-only and
  contexts shorter than the windows;
* the fused decode step with windows, end to end;
* folded value rotation with windows, and an out-of-range window slot.
"""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_02691_gb300 import optr, synth

import parity_helpers as ph

pytestmark = pytest.mark.gpu

VARIANTS = [optr.OPTR_VARIANT_CUDA_CORE, optr.OPTR_VARIANT_TENSOR]
# long128k: one sequence, so the combine splits each (sequence, KV head)
# over several CTAs (the last one merges the window partials)
CASES = [("tiny", 1.0), ("decode8k", 1 / 16), ("ragged", 1 / 32),
         ("long128k", 1 / 32)]
WINDOWS = [(64, 256), (16, 32), (0, 48), (32, 0)]


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


def _case(name, scale, sink, recent, seed=0):
    """Workload plus its oracle state: pool, pre-rounding values and the
    window store (slots a permutation, two spare slots)."""
    key = (name, scale, sink, recent, seed)
    if key not in _cache:
        c = synth.build_case(synth.workload(name, seed, scale), seed)
        pool, u_ctx, u_new = ph.oracle_case(c)
        n_slots = c["B"] + 2
        slots = np.random.default_rng(seed + 5).permutation(n_slots)[:c["B"]]
        slots = slots.astype(np.int32)
        win = oracle.new_windows(n_slots, c["h_kv"], sink, recent)
        for kk, vv, cu, pos0 in ((c["k_ctx"], c["v_ctx"], c["cu_ctx"], c["pos0_ctx"]),
                                 (c["k_new"], c["v_new"], c["cu_new"], c["pos0_new"])):
            if kk.shape[0]:
                oracle.window_write(synth.bf16_bits(kk), synth.bf16_bits(vv),
                                    cu.numpy(), pos0.numpy(), win, slots, sink,
                                    recent)
        _cache[key] = (c, pool, u_ctx, u_new, win, slots)
    return _cache[key]


def _oracle_decode(c, pool, win, slots, sink, recent, R_v=None):
    return oracle.decode_attention(
        synth.bf16_bits(c["q"]), c["block_table"].numpy(),
        c["seq_lens"].numpy(), pool, c["R_k"].numpy(),
        (c["R_v"] if R_v is None else R_v).numpy(), c["h_kv"], win=win,
        win_slot=slots, sink=sink, recent=recent, mu=c["mu"].numpy())


def _win_tensor(win_np, dev="cuda"):
    return torch.from_numpy(win_np.view(np.int16)).view(torch.bfloat16).to(dev)


def _gpu_run(c, sink, recent, slots, n_slots, avar=0, dvar=0, step=True,
             R_v="given", dev="cuda"):
    p = optr.optr_params_create(c["R_k"], c["R_v"] if R_v == "given" else R_v,
                                c["mu"], c["h_q"], append_variant=avar,
                                decode_variant=dvar, sink=sink, recent=recent)
    pool = optr.new_pool(p, c["num_pages"], device=dev)
    win = optr.new_windows(p, n_slots, device=dev)
    ws_slot = torch.from_numpy(slots).to(dev)
    bt = c["block_table"].to(dev)
    optr.optr_kv_append_win(p, c["k_ctx"].to(dev), c["v_ctx"].to(dev),
                            c["cu_ctx"].to(dev), c["pos0_ctx"].to(dev), bt,
                            pool, win, ws_slot)
    out = torch.full((c["B"], c["h_q"], 128), 7.0, dtype=torch.float32,
                     device=dev)
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device=dev)
    if step and c["k_new"].shape[0]:
        optr.optr_decode_step_win(p, c["q"].to(dev), c["k_new"].to(dev),
                                  c["v_new"].to(dev), c["cu_new"].to(dev),
                                  c["pos0_new"].to(dev), bt,
                                  c["seq_lens"].to(dev), pool, win, ws_slot,
                                  out, ws)
    else:
        if c["k_new"].shape[0]:
            optr.optr_kv_append_win(p, c["k_new"].to(dev), c["v_new"].to(dev),
                                    c["cu_new"].to(dev), c["pos0_new"].to(dev),
                                    bt, pool, win, ws_slot)
        optr.optr_decode_attention_win(p, c["q"].to(dev), bt,
                                       c["seq_lens"].to(dev), pool, win,
                                       ws_slot, out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    return p, pool, win, out


def _win_bits(win):
    return win.cpu().view(torch.int16).numpy().view(np.uint16)


@pytest.mark.parametrize("name,scale", CASES)
@pytest.mark.parametrize("avar", VARIANTS)
@pytest.mark.parametrize("step", [False, True])
def test_window_cache_write(name, scale, avar, step):
    """INT2 records as without windows; the store bit-exact."""
    sink, recent = 64, 256
    c, pool_ref, u_ctx, u_new, win_ref, slots = _case(name, scale, sink, recent)
    _, pool, win, _ = _gpu_run(c, sink, recent, slots, win_ref.shape[0],
                               avar=avar, step=step)
    np.testing.assert_array_equal(_win_bits(win), win_ref)
    pg = pool.cpu().numpy()
    for cu, pos0, u in ((c["cu_ctx"], c["pos0_ctx"], u_ctx),
                        (c["cu_new"], c["pos0_new"], u_new)):
        if u is None:
            continue
        pages, slots_ = ph.token_slots(cu, pos0, c["block_table"])
        ph.compare_append(pg, pool_ref, u, pages, slots_)


@pytest.mark.parametrize("name,scale", CASES)
@pytest.mark.parametrize("sink,recent", WINDOWS)
@pytest.mark.parametrize("dvar", VARIANTS)
def test_window_decode(name, scale, sink, recent, dvar):
    """Decode over the oracle's pool and store, against the oracle."""
    c, pool_ref, _, _, win_ref, slots = _case(name, scale, sink, recent)
    dev = "cuda"
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                decode_variant=dvar, sink=sink, recent=recent)
    pool = torch.from_numpy(pool_ref).to(dev)
    win = _win_tensor(win_ref)
    bt = c["block_table"].to(dev)
    out = torch.full((c["B"], c["h_q"], 128), 7.0, dtype=torch.float32,
                     device=dev)
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device=dev)
    optr.optr_decode_attention_win(p, c["q"].to(dev), bt, c["seq_lens"].to(dev),
                                   pool, win, torch.from_numpy(slots).to(dev),
                                   out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    ref = _oracle_decode(c, pool_ref, win_ref, slots, sink, recent)
    e = ph.assert_decode_close(out.cpu().double().numpy(), ref,
                               f"{name} windows ({sink}, {recent})")
    print(f"{name} ({sink}, {recent}) variant {dvar}: err/rms {e:.2e}")


@pytest.mark.parametrize("dvar", VARIANTS)
def test_window_decode_short_and_empty_sequences(dvar):
    """Sequences shorter than the sink, inside the windows, just past them,
    and empty; one sequence of several thousand tokens in the same batch."""
    sink, recent = 64, 256
    lens = [0, 1, 17, 64, 65, 200, 320, 321, 337, 4000]
    B, h_kv, h_q = len(lens), 8, 32
    seed = 9
    n = sum(lens)
    k, v = synth.kv_tokens(n, h_kv, "t4", seed, 0)
    mu = synth.key_mean(k)
    R_k, R_v = synth.rotations(h_kv, seed)
    q = synth.queries(B, h_q, seed)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    bt, num_pages = synth.page_tables([max(x, 1) for x in lens], True, seed)
    pool_ref = np.zeros((num_pages, h_kv, 1536), np.uint8)
    oracle.kv_append(synth.bf16_bits(k), synth.bf16_bits(v), cu,
                     np.zeros(B, np.int32), bt.numpy(), pool_ref, R_k.numpy(),
                     R_v.numpy(), mu.numpy())
    slots = np.arange(B, dtype=np.int32)[::-1].copy()
    win_ref = oracle.new_windows(B, h_kv, sink, recent)
    oracle.window_write(synth.bf16_bits(k), synth.bf16_bits(v), cu,
                        np.zeros(B, np.int32), win_ref, slots, sink, recent)
    c = dict(q=q, block_table=bt, seq_lens=torch.tensor(lens, dtype=torch.int32),
             R_k=R_k, R_v=R_v, mu=mu, h_kv=h_kv)
    ref = _oracle_decode(c, pool_ref, win_ref, slots, sink, recent)
    p = optr.optr_params_create(R_k, R_v, mu, h_q, decode_variant=dvar,
                                sink=sink, recent=recent)
    out = torch.full((B, h_q, 128), 7.0, dtype=torch.float32, device="cuda")
    ws = optr.new_workspace(p, B, bt.shape[1], device="cuda")
    optr.optr_decode_attention_win(p, q.cuda(), bt.cuda(), c["seq_lens"].cuda(),
                                   torch.from_numpy(pool_ref).cuda(),
                                   _win_tensor(win_ref),
                                   torch.from_numpy(slots).cuda(), out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    got = out.cpu().double().numpy()
    assert not got[0].any()
    ph.assert_decode_close(got[1:], ref[1:], "short sequences")


@pytest.mark.parametrize("name,scale", CASES)
@pytest.mark.parametrize("dvar", VARIANTS)
def test_window_step_end_to_end(name, scale, dvar):
    """GPU cache write and decode step with windows against the oracle's,
    every row asserted at OUT_TOL * RMS plus the perturbation bound of the
    INT2 records that differ within the append tolerance (0 when none)."""
    sink, recent = 64, 256
    c, pool_ref, u_ctx, u_new, win_ref, slots = _case(name, scale, sink, recent)
    _, pool, win, out = _gpu_run(c, sink, recent, slots, win_ref.shape[0],
                                 dvar=dvar, step=True)
    np.testing.assert_array_equal(_win_bits(win), win_ref)
    pg = pool.cpu().numpy()
    diffs = []
    for cu, pos0, u in ((c["cu_ctx"], c["pos0_ctx"], u_ctx),
                        (c["cu_new"], c["pos0_new"], u_new)):
        if u is None:
            continue
        pages, slots_ = ph.token_slots(cu, pos0, c["block_table"])
        st = ph.compare_append(pg, pool_ref, u, pages, slots_)
        diffs.append((cu.numpy(), pos0.numpy(), st["flipped"]))
    got = out.cpu().double().numpy()
    ref = _oracle_decode(c, pool_ref, win_ref, slots, sink, recent)
    bound = ph.e2e_row_bounds(c, pool_ref, pg, diffs, win=win_ref,
                              win_slot=slots, sink=sink, recent=recent)
    strict, mean_bar = ph.assert_rows_within_bar(got, ref, bound,
                                                 f"{name} step windows")
    print(f"{name} windows variant {dvar}: strict rows {strict:.2f}, mean bar "
          f"{mean_bar:.3f} x strict")


def test_window_step_equals_append_then_decode():
    """The fused step (window copies in the prologue launch) gives the bytes
    and output of the two separate calls."""
    sink, recent = 64, 256
    c, _, _, _, win_ref, slots = _case("decode8k", 1 / 16, sink, recent)
    r = [_gpu_run(c, sink, recent, slots, win_ref.shape[0], step=s)
         for s in (False, True)]
    assert torch.equal(r[0][1], r[1][1])
    assert torch.equal(r[0][2], r[1][2])
    assert torch.equal(r[0][3], r[1][3])


def test_window_folded_value_rotation():
    """R_v = NULL with windows: the oracle with R_v = I."""
    sink, recent = 64, 256
    c0 = synth.build_case(synth.workload("ragged", 0, 1 / 32), 0)
    eye = torch.eye(128).expand(c0["h_kv"], 128, 128).contiguous()
    c = dict(c0)
    c["R_v"] = eye
    pool_ref, _, _ = ph.oracle_case(c)
    n_slots = c["B"]
    slots = np.arange(n_slots, dtype=np.int32)
    win_ref = oracle.new_windows(n_slots, c["h_kv"], sink, recent)
    for kk, vv, cu, pos0 in ((c["k_ctx"], c["v_ctx"], c["cu_ctx"], c["pos0_ctx"]),
                             (c["k_new"], c["v_new"], c["cu_new"], c["pos0_new"])):
        oracle.window_write(synth.bf16_bits(kk), synth.bf16_bits(vv), cu.numpy(),
                            pos0.numpy(), win_ref, slots, sink, recent)
    for dvar in VARIANTS:
        p = optr.optr_params_create(c["R_k"], None, c["mu"], c["h_q"],
                                    decode_variant=dvar, sink=sink,
                                    recent=recent)
        bt = c["block_table"].cuda()
        out = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32,
                          device="cuda")
        ws = optr.new_workspace(p, c["B"], bt.shape[1], device="cuda")
        optr.optr_decode_attention_win(p, c["q"].cuda(), bt,
                                       c["seq_lens"].cuda(),
                                       torch.from_numpy(pool_ref).cuda(),
                                       _win_tensor(win_ref),
                                       torch.from_numpy(slots).cuda(), out, ws)
        torch.cuda.synchronize()
        assert optr.optr_device_error(p) == 0
        ref = _oracle_decode(c, pool_ref, win_ref, slots, sink, recent, R_v=eye)
        ph.assert_decode_close(out.cpu().double().numpy(), ref, "folded windows")


def test_window_slot_out_of_range_is_flagged():
    """A window slot outside [0, n_slots) skips that sequence's window work
    (nothing read or written there) and sets OPTR_DEVERR_WIN_SLOT; the
    other sequences are unaffected."""
    sink, recent = 64, 256
    c, pool_ref, _, _, win_ref, slots = _case("decode8k", 1 / 16, sink, recent)
    bad = slots.copy()
    bad[3] = win_ref.shape[0] + 5
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                sink=sink, recent=recent)
    bt = c["block_table"].cuda()
    out = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device="cuda")
    ws = optr.new_workspace(p, c["B"], bt.shape[1], device="cuda")
    optr.optr_decode_attention_win(p, c["q"].cuda(), bt, c["seq_lens"].cuda(),
                                   torch.from_numpy(pool_ref).cuda(),
                                   _win_tensor(win_ref),
                                   torch.from_numpy(bad).cuda(), out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == optr.OPTR_DEVERR_WIN_SLOT
    ref = _oracle_decode(c, pool_ref, win_ref, slots, sink, recent)
    got = out.cpu().double().numpy()
    keep = np.arange(c["B"]) != 3
    ph.assert_decode_close(got[keep], ref[keep], "other sequences")
    assert np.all(np.isfinite(got))


@pytest.mark.parametrize("dvar", VARIANTS)
def test_window_decode_many_sequences(dvar):
    """300 sequences (more than the partial kernel caches page prefix sums
    for, so it reads them after waiting), lengths from 1 to 700."""
    sink, recent = 64, 256
    g = np.random.default_rng(13)
    lens = g.integers(1, 700, size=300).tolist()
    B, h_kv, h_q = len(lens), 8, 32
    k, v = synth.kv_tokens(sum(lens), h_kv, "t4", 13, 0)
    mu = synth.key_mean(k)
    R_k, R_v = synth.rotations(h_kv, 13)
    q = synth.queries(B, h_q, 13)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    bt, num_pages = synth.page_tables(lens, True, 13)
    pool_ref = np.zeros((num_pages, h_kv, 1536), np.uint8)
    oracle.kv_append(synth.bf16_bits(k), synth.bf16_bits(v), cu,
                     np.zeros(B, np.int32), bt.numpy(), pool_ref, R_k.numpy(),
                     R_v.numpy(), mu.numpy())
    slots = g.permutation(B + 7)[:B].astype(np.int32)
    win_ref = oracle.new_windows(B + 7, h_kv, sink, recent)
    oracle.window_write(synth.bf16_bits(k), synth.bf16_bits(v), cu,
                        np.zeros(B, np.int32), win_ref, slots, sink, recent)
    c = dict(q=q, block_table=bt, seq_lens=torch.tensor(lens, dtype=torch.int32),
             R_k=R_k, R_v=R_v, mu=mu, h_kv=h_kv)
    ref = _oracle_decode(c, pool_ref, win_ref, slots, sink, recent)
    p = optr.optr_params_create(R_k, R_v, mu, h_q, decode_variant=dvar,
                                sink=sink, recent=recent)
    out = torch.full((B, h_q, 128), 7.0, dtype=torch.float32, device="cuda")
    ws = optr.new_workspace(p, B, bt.shape[1], device="cuda")
    optr.optr_decode_attention_win(p, q.cuda(), bt.cuda(), c["seq_lens"].cuda(),
                                   torch.from_numpy(pool_ref).cuda(),
                                   _win_tensor(win_ref),
                                   torch.from_numpy(slots).cuda(), out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    ph.assert_decode_close(out.cpu().double().numpy(), ref, "300 sequences")


def test_plain_entry_points_reject_windows():
    c = synth.build_case(synth.workload("tiny", 0, 1 / 16), 0)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                sink=64, recent=256)
    pool = optr.new_pool(p, c["num_pages"])
    with pytest.raises(optr.OptrError):
        optr.optr_kv_append(p, c["k_ctx"].cuda(), c["v_ctx"].cuda(),
                            c["cu_ctx"].cuda(), c["pos0_ctx"].cuda(),
                            c["block_table"].cuda(), pool)


def test_window_step_replays_from_a_cuda_graph():
    """The windowed decode step (window copy CTAs in the prologue launch,
    window warps in the partial kernel, window merge in the combine)
    captured once in a CUDA graph and replayed gives the bytes and output of
    a direct call."""
    sink, recent = 64, 256
    c, _, _, _, win_ref, slots = _case("decode8k", 1 / 16, sink, recent)
    dev = "cuda"
    res = []
    for use_graph in (False, True):
        p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], c["h_q"],
                                    sink=sink, recent=recent)
        pool = optr.new_pool(p, c["num_pages"], device=dev)
        win = optr.new_windows(p, win_ref.shape[0], device=dev)
        ws_slot = torch.from_numpy(slots).to(dev)
        bt = c["block_table"].to(dev)
        optr.optr_kv_append_win(p, c["k_ctx"].to(dev), c["v_ctx"].to(dev),
                                c["cu_ctx"].to(dev), c["pos0_ctx"].to(dev), bt,
                                pool, win, ws_slot)
        args = [c["q"].to(dev), c["k_new"].to(dev), c["v_new"].to(dev),
                c["cu_new"].to(dev), c["pos0_new"].to(dev), bt,
                c["seq_lens"].to(dev), pool, win, ws_slot]
        out = torch.empty(c["B"], c["h_q"], 128, dtype=torch.float32, device=dev)
        ws = optr.new_workspace(p, c["B"], bt.shape[1], device=dev)
        torch.cuda.synchronize()
        if use_graph:
            s = torch.cuda.Stream()
            s.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(s):  # warm-up outside the capture
                optr.optr_decode_step_win(p, *args, out, ws)
            torch.cuda.current_stream().wait_stream(s)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                optr.optr_decode_step_win(p, *args, out, ws)
            out.zero_()
            g.replay()
        else:
            optr.optr_decode_step_win(p, *args, out, ws)
            optr.optr_decode_step_win(p, *args, out, ws)
        torch.cuda.synchronize()
        assert optr.optr_device_error(p) == 0
        res.append((pool.cpu(), win.cpu(), out.cpu()))
    for a, b in zip(*res):
        assert torch.equal(a, b)


def test_long_write_copies_only_window_rows():
    """A write of several thousand tokens per sequence in one call (the
    prefill case: tiles of 256 tokens with few window rows each) fills the
    store exactly as the oracle's rule."""
    sink, recent = 64, 256
    lens = [3000, 64, 700, 1, 2500]
    B, h_kv = len(lens), 8
    k, v = synth.kv_tokens(sum(lens), h_kv, "t4", 5, 0)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    pos0 = np.array([0, 10, 300, 5000, 40], np.int32)
    slots = np.array([4, 0, 3, 1, 2], np.int32)
    win_ref = oracle.new_windows(B, h_kv, sink, recent)
    oracle.window_write(synth.bf16_bits(k), synth.bf16_bits(v), cu, pos0,
                        win_ref, slots, sink, recent)
    R_k, R_v = synth.rotations(h_kv, 5)
    p = optr.optr_params_create(R_k, R_v, synth.key_mean(k), 32, sink=sink,
                                recent=recent)
    total = [int(a) + int(b) for a, b in zip(pos0, lens)]
    bt, num_pages = synth.page_tables(total, True, 5)
    pool = optr.new_pool(p, num_pages)
    win = optr.new_windows(p, B)
    optr.optr_kv_append_win(p, k.cuda(), v.cuda(), torch.from_numpy(cu).cuda(),
                            torch.from_numpy(pos0).cuda(), bt.cuda(), pool, win,
                            torch.from_numpy(slots).cuda())
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    np.testing.assert_array_equal(_win_bits(win), win_ref)
