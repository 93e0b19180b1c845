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
    """codes [n][h_kv][128] and (scale, min) float64 [n][h_kv][4] (the
    compact G = 128 record's one pair repeated in the four entries; the
    pool's record size, 1536 or 1152 bytes, gives its layout)."""
    chunk = pool[pages]  # [n, h_kv, 1536 or 1152]
    compact = pool.shape[-1] == 1152
    off = 512 * kind
    idx = off + slots[:, None] * 32 + np.arange(32)[None]
    cb = np.take_along_axis(chunk, idx[:, None, :].repeat(chunk.shape[1], 1), 2)
    codes = (cb[..., CODE_BYTE] >> CODE_SHIFT) & 3
    if compact:
        moff = 1024 + 64 * kind
        midx = moff + slots[:, None] * 4 + np.tile(np.arange(4), 4)[None]
    else:
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
    """GPU decode over a given (oracle-written) host pool (its record size,
    1536 or 1152 bytes, selects the G = 32 or the compact G = 128 layout)."""
    group = 128 if pool_np.shape[-1] == 1152 else 32
    p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                case["h_q"], decode_variant=variant, group=group)
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


def oracle_case(case, pool_init=None, group=32, clip_k=1.0, clip_v=1.0):
    """Oracle append of context and new tokens; returns (pool, u_ctx, u_new)."""
    pool = (np.zeros((case["num_pages"], case["h_kv"], oracle.chunk_bytes(group)),
                     np.uint8)
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


def dequant_records(pool, pages, slots, h, kind):
    """Dequantized rotated vectors code * scale + min (float64 [n][128]) of
    KV head h at the given (page, slot) records of a pool; kind 0 = keys,
    1 = values (slot_codes repeats a compact record's pair per 32-channel
    block, so one reading serves both layouts)."""
    codes, sc, mn = slot_codes(pool, pages, slots, kind)
    grp = _CH // 32
    return codes[:, h, :] * sc[:, h, grp] + mn[:, h, grp]


def e2e_row_bounds(case, pool_ref, pool_gpu, diffs, win=None, win_slot=None,
                   sink=0, recent=0):
    """Per output row, how far exact attention over the GPU-written cache may
    lie from exact attention over the oracle-written one, given where the
    two caches differ (in-band codes, an fp16 ulp of scale or min: both
    within the append tolerance).  ``diffs`` is a list of (cu, pos0,
    mask[n_tok][h_kv]) marking the differing token records of each write.
    With BF16 windows (``win``: the oracle's store, bf16 bits
    [n_slots][h_kv][2][sink + recent][128]; ``win_slot`` [B]) window
    positions are read from the store, so their pool records never count.

    For a row (b, j) of KV head h let D be the INT2 positions whose records
    differ, p the oracle's softmax weights over the oracle cache, delta_s =
    q'_j . (k'_s - k_s) / sqrt(d) the logit change (Sec. 3 Eq. 1 in the
    rotated basis, Appendix "Rotated-query implementation") and
    dv_s = v'_s - v_s.  The weights over the GPU cache are
    p'_s = p_s e^{delta_s} / Z with Z = 1 + sum_D p_s (e^{delta_s} - 1), so,
    with every value taken in the output basis (v R_v^T for INT2 positions,
    the stored bf16 value for window positions),

      |o' - o|_2 <= sum_D p'_s |dv_s|_2
                    + (sum_s |p'_s - p_s|) * max_s |v_s - o|_2,
      sum_s |p'_s - p_s| = ((1 - P_D)|1 - Z| + sum_D p_s |e^{delta_s} - Z|) / Z,

    exactly (Sec. 3 Eq. 2; the sum of p' - p is zero, so any centre may be
    subtracted from v; R_v is orthogonal, so |dv R_v^T|_2 = |dv|_2), and
    |x|_inf <= |x|_2 bounds every element of the row.  Rows of groups with
    no differing record get 0."""
    B, h_q, h_kv = case["B"], case["h_q"], case["h_kv"]
    ratio = h_q // h_kv
    bt = case["block_table"].numpy()
    lens = case["seq_lens"].numpy()
    R_k = case["R_k"].numpy().astype(np.float64)
    R_v = case["R_v"].numpy().astype(np.float64)
    q = case["q"].float().numpy().astype(np.float64)
    windows = sink > 0 or recent > 0
    where = {}
    for cu, pos0, mask in diffs:
        cu = np.asarray(cu)
        pos0 = np.asarray(pos0)
        for t, h in np.argwhere(mask):
            b = int(np.searchsorted(cu, t, side="right") - 1)
            where.setdefault((b, int(h)), set()).add(int(pos0[b] + t - cu[b]))
    bound = np.zeros((B, h_q))
    for (b, h), poss in sorted(where.items()):
        n = int(lens[b])
        allp = np.arange(n)
        in_win = (allp < sink) | (allp >= n - recent) if windows else np.zeros(n, bool)
        d = np.array(sorted(s for s in poss if s < n and not in_win[s]), np.int64)
        if n == 0 or d.size == 0:
            continue
        kr = dequant_records(pool_ref, bt[b, allp // 16], allp % 16, h, 0)
        vr = dequant_records(pool_ref, bt[b, allp // 16], allp % 16, h, 1)
        dk = dequant_records(pool_gpu, bt[b, d // 16], d % 16, h, 0) - kr[d]
        dv = dequant_records(pool_gpu, bt[b, d // 16], d % 16, h, 1) - vr[d]
        dvn = np.linalg.norm(dv, axis=1)
        vout = vr @ R_v[h].T  # output basis
        if windows:
            wp = allp[in_win]
            rows = np.where(wp < sink, wp, sink + (wp - sink) % max(recent, 1))
            bits = np.asarray(win)[int(win_slot[b]), h, 1, rows, :]
            vout[in_win] = (bits.astype(np.uint32) << 16).view(np.float32)
        for r in range(ratio):
            j = ratio * h + r
            _, p = oracle.decode_attention(
                synth.bf16_bits(case["q"]), bt, lens, pool_ref,
                case["R_k"].numpy(), case["R_v"].numpy(), h_kv,
                rows=[(b, j)], want_p=True, win=win, win_slot=win_slot,
                sink=sink, recent=recent,
                mu=case["mu"].numpy() if windows else None)
            qp = (q[b, j] @ R_k[h]) / np.sqrt(128.0)
            a = np.exp(dk @ qp)
            pd = p[d]
            Z = 1.0 + float(np.sum(pd * (a - 1.0)))
            term_v = float(np.sum(pd * a / Z * dvn))
            o = p @ vout
            spread = float(np.max(np.linalg.norm(vout - o, axis=1)))
            dp = ((1.0 - pd.sum()) * abs(1.0 - Z) +
                  float(np.sum(pd * np.abs(a - Z)))) / Z
            bound[b, j] = term_v + dp * spread
    return bound


def assert_rows_within_bar(got, ref, bound, what=""):
    """Every row: max |gpu - oracle| <= OUT_TOL * RMS(oracle) + bound(row).
    Returns (share of rows checked at the strict bar, mean bar / strict)."""
    rms = float(np.sqrt(np.mean(ref ** 2)))
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    bar = OUT_TOL * rms + bound
    err = np.abs(got - ref).max(axis=2)
    worst = np.unravel_index(np.argmax(err / bar), err.shape)
    assert np.all(err <= bar * (1 + 1e-9)), (
        f"{what}: row {worst} err {err[worst]:.3e} > bar {bar[worst]:.3e} "
        f"(bound {bound[worst]:.3e}, strict {OUT_TOL * rms:.3e})")
    return float((bound == 0).mean()), float(bar.mean() / (OUT_TOL * rms))
