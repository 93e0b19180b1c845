"""Helpers for the GPU-vs-oracle parity tests (imported by test_gpu_*.py).

Tolerances (stated once, used by every parity test):
  codes       bit-exact, except codes whose oracle pre-rounding value u lies
              within TIE_BAND of a rounding boundary 0.5 / 1.5 / 2.5
              (those are counted and reported);
  scale, min  |gpu - oracle| <= META_RTOL * max(|oracle|, oracle scale);
  decode      max |gpu - oracle| <= OUT_TOL * RMS(oracle output).
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import oracle
from paper_2608_02691_gb300 import optr, synth

TIE_BAND = 1e-5
META_RTOL = 1e-3
OUT_TOL = 2e-3

_CH = np.arange(128)
# layout of a slot's code bytes (include/optr.h): ch = 32g + 4w + r at byte
# 4w + g, bits [2r, 2r+1]
CODE_BYTE = 4 * ((_CH % 32) // 4) + _CH // 32
CODE_SHIFT = 2 * (_CH % 4)


def token_slots(cu, pos0, bt):
    """(physical page, slot) of every appended token."""
    cu = np.asarray(cu)
    pos0 = np.asarray(pos0)
    bt = np.asarray(bt)
    pages, slots = [], []
    for b in range(len(pos0)):
        for t in range(cu[b], cu[b + 1]):
            pos = pos0[b] + t - cu[b]
            pages.append(bt[b, pos // 16])
            slots.append(pos % 16)
    return np.array(pages, np.int64), np.array(slots, np.int64)


def slot_codes(pool, pages, slots, kind):
    """codes [n][h_kv][128] and (scale, min) float64 [n][h_kv][4]."""
    chunk = pool[pages]  # [n, h_kv, 1536]
    off = 512 * kind
    idx = off + slots[:, None] * 32 + np.arange(32)[None]
    cb = np.take_along_axis(chunk, idx[:, None, :].repeat(chunk.shape[1], 1), 2)
    codes = (cb[..., CODE_BYTE] >> CODE_SHIFT) & 3
    moff = 1024 + 256 * kind
    midx = moff + slots[:, None] * 16 + np.arange(16)[None]
    mb = np.take_along_axis(chunk, midx[:, None, :].repeat(chunk.shape[1], 1), 2)
    meta = np.ascontiguousarray(mb).view(np.float16).astype(np.float64)
    return codes, meta[..., 0::2], meta[..., 1::2]


def compare_append(pool_gpu, pool_ref, u, pages, slots):
    """Returns a dict of counts (and the boolean [n_tok][h_kv] mask of
    token-heads whose stored record differs within tolerance -- an in-band
    code or a scale/min ulp -- under key "flipped");
    raises AssertionError on a violation."""
    stats = {"codes": 0, "tie_band": 0, "mismatch_in_band": 0,
             "flipped": np.zeros(u.shape[:2], bool)}
    for kind in (0, 1):
        cg, sg, mg = slot_codes(pool_gpu, pages, slots, kind)
        cr, sr, mr = slot_codes(pool_ref, pages, slots, kind)
        uu = u[:, :, kind, :]
        fl = np.floor(uu)
        band = (np.abs(uu - fl - 0.5) < TIE_BAND) & (fl >= 0) & (fl <= 2)
        bad = (cg != cr) & ~band
        stats["codes"] += cg.size
        stats["tie_band"] += int(band.sum())
        stats["mismatch_in_band"] += int(((cg != cr) & band).sum())
        stats["flipped"] |= ((cg != cr) & band).any(axis=2)
        # an in-tolerance fp16 ulp of scale or min also changes the output
        stats["flipped"] |= ((sg != sr) | (mg != mr)).any(axis=2)
        if bad.any():
            i = np.argwhere(bad)[0]
            raise AssertionError(
                f"kind {kind}: {int(bad.sum())} code mismatches outside the tie "
                f"band; first at token {i[0]} head {i[1]} ch {i[2]}: gpu "
                f"{cg[tuple(i)]} oracle {cr[tuple(i)]} u {uu[tuple(i)]}")
        tol_s = META_RTOL * np.maximum(np.abs(sr), 1e-30)
        assert np.all(np.abs(sg - sr) <= tol_s + 1e-12), f"kind {kind} scale"
        tol_m = META_RTOL * np.maximum(np.abs(mr), sr)
        assert np.all(np.abs(mg - mr) <= tol_m + 1e-12), f"kind {kind} min"
    return stats


def assert_decode_close(got, ref, what=""):
    rms = float(np.sqrt(np.mean(ref ** 2)))
    err = float(np.abs(got - ref).max())
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    assert err <= OUT_TOL * rms, f"{what}: max|err| {err:.3e} > {OUT_TOL} * rms {rms:.3e}"
    return err / max(rms, 1e-300)


def gpu_case(case, variant=optr.OPTR_VARIANT_DEFAULT, append_variant=0,
             poison=False, dev="cuda"):
    """Run append (context, then the step's new tokens) and decode on the GPU.
    Returns (params, pool tensor, out tensor)."""
    p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                case["h_q"], decode_variant=variant,
                                append_variant=append_variant)
    pool = optr.new_pool(p, case["num_pages"], device=dev)
    if poison:
        pool.fill_(0xFF)  # NaN metadata in every slot not written below
    bt = case["block_table"].to(dev)
    if case["k_ctx"].shape[0]:
        optr.optr_kv_append(p, case["k_ctx"].to(dev), case["v_ctx"].to(dev),
                            case["cu_ctx"].to(dev), case["pos0_ctx"].to(dev),
                            bt, pool)
    if case["k_new"].shape[0]:
        optr.optr_kv_append(p, case["k_new"].to(dev), case["v_new"].to(dev),
                            case["cu_new"].to(dev), case["pos0_new"].to(dev),
                            bt, pool)
    out = torch.empty(case["B"], case["h_q"], 128, dtype=torch.float32,
                      device=dev)
    ws = optr.new_workspace(p, case["B"], bt.shape[1], device=dev)
    optr.optr_decode_attention(p, case["q"].to(dev), bt,
                               case["seq_lens"].to(dev), pool, out, ws)
    torch.cuda.synchronize()
    return p, pool, out


def gpu_decode(case, pool_np, variant=optr.OPTR_VARIANT_DEFAULT,
               seq_lens=None, dev="cuda"):
    """GPU decode over a given (oracle-written) host pool."""
    p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                case["h_q"], decode_variant=variant)
    pool = torch.from_numpy(pool_np).to(dev)
    bt = case["block_table"].to(dev)
    lens = case["seq_lens"] if seq_lens is None else seq_lens
    out = torch.full((case["B"], case["h_q"], 128), 7.0, dtype=torch.float32,
                     device=dev)
    ws = optr.new_workspace(p, case["B"], bt.shape[1], device=dev)
    optr.optr_decode_attention(p, case["q"].to(dev), bt, lens.to(dev), pool,
                               out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    return out.cpu().double().numpy()


def flipped_groups(case, stats_ctx, stats_new):
    """(b, h) groups whose cached codes differ in the tie band somewhere."""
    out = set()
    for st, cu in ((stats_ctx, case["cu_ctx"]), (stats_new, case["cu_new"])):
        if st is None:
            continue
        cu = np.asarray(cu)
        for t, h in np.argwhere(st["flipped"]):
            b = int(np.searchsorted(cu, t, side="right") - 1)
            out.add((b, int(h)))
    return out


def oracle_case(case, pool_init=None, group=32, clip_k=1.0, clip_v=1.0):
    """Oracle append of context and new tokens; returns (pool, u_ctx, u_new)."""
    pool = (np.zeros((case["num_pages"], case["h_kv"], 1536), np.uint8)
            if pool_init is None else pool_init.copy())
    bt = case["block_table"].numpy()
    args = (case["R_k"].numpy(), case["R_v"].numpy(), case["mu"].numpy())
    u_ctx = u_new = None
    if case["k_ctx"].shape[0]:
        u_ctx = oracle.kv_append(synth.bf16_bits(case["k_ctx"]),
                                 synth.bf16_bits(case["v_ctx"]),
                                 case["cu_ctx"].numpy(),
                                 case["pos0_ctx"].numpy(), bt, pool, *args,
                                 want_u=True, group=group, clip_k=clip_k,
                                 clip_v=clip_v)
    if case["k_new"].shape[0]:
        u_new = oracle.kv_append(synth.bf16_bits(case["k_new"]),
                                 synth.bf16_bits(case["v_new"]),
                                 case["cu_new"].numpy(),
                                 case["pos0_new"].numpy(), bt, pool, *args,
                                 want_u=True, group=group, clip_k=clip_k,
                                 clip_v=clip_v)
    return pool, u_ctx, u_new


def oracle_decode(case, pool, rows=None, seq_lens=None, q=None):
    return oracle.decode_attention(
        synth.bf16_bits(case["q"] if q is None else q),
        case["block_table"].numpy(),
        (case["seq_lens"] if seq_lens is None else seq_lens).numpy(), pool,
        case["R_k"].numpy(), case["R_v"].numpy(), case["h_kv"], rows=rows)
