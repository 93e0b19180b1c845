"""Benchmark of the rotated INT2 paged KV-cache hot path on one GB300.

One step = one decode step of the Qwen3-8B-shaped layer (batch 16, 32 query /
8 KV heads, head dim 128, context 8192 per sequence, page size 16, shuffled
pages): append the step's new token of every sequence (center, rotate,
INT2-quantize, pack, scatter) and run decode attention over the 8193 cached
tokens (rotate queries, stream the INT2 pages, split-K online softmax,
combine, apply R_v^T).  The cache is pre-filled by the library's append
before timing.  Metric: algorithmic HBM bytes of the step per second (codes
and fp16 scale/min read, bf16 query read, fp32 output written, plus the
appended token's bf16 K/V read and INT2 record written).

Extra measurements in the same JSON line: the prefill append workload
(4 x 32768 tokens) in tokens/s, the long-context (131072) and ragged
(batch 128) decode workloads, and the CPU oracle on a bounded sample.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
Multi-GPU (weak scaling, no data-path collective): torchrun ... bench.py --gpus N.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

D = 128
CHUNK = 1536
L2_FLUSH_BYTES = 512 << 20


# ------------------------------------------------------------------ utils

def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during timing."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index),
                 f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        time.sleep(0.3)

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], 0.0, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap")
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax = max(smax, float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": smax,
                "samples": len(sm), "reasons": sorted(reasons)}


def kernel_source_hash(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2608_02691_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def traffic_for(kernel_key, files):
    """dram bytes per launch from the committed ncu summary, if the kernel's
    source is unchanged since the counters were taken (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        e = d[kernel_key]
        if e.get("source_sha") == kernel_source_hash(files):
            return float(e["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


# ------------------------------------------------------------ byte counts

def record_bytes(group=32):
    """Cache bytes per token and KV head: 32 + 32 code bytes and 16 + 16
    metadata bytes (G = 32), or 4 + 4 metadata bytes (the compact G = 128
    record)."""
    return 72 if group == 128 else 96


def decode_bytes(seq_lens, h_kv, h_q, group=32):
    """Algorithmic bytes of one decode: the cache records of every cached
    token and KV head, bf16 query, fp32 output."""
    toks = int(sum(int(x) for x in seq_lens))
    B = len(seq_lens)
    return toks * h_kv * record_bytes(group) + B * h_q * D * 2 + B * h_q * D * 4


def decode_stream_bytes(seq_lens, h_kv):
    """Bytes the split-K partial kernel streams: codes + metadata only."""
    return int(sum(int(x) for x in seq_lens)) * h_kv * 96


def append_bytes(n_tok, h_kv, group=32):
    """Append: bf16 K and V read (512 B) + the record written per token and
    head."""
    return n_tok * h_kv * (512 + record_bytes(group))


def window_split(n, sink, recent):
    """(INT2 tokens, BF16 window tokens) of a sequence of n tokens: window
    positions are s < sink and s >= n - recent."""
    ns = min(n, sink)
    r0 = max(sink, n - recent)
    nw = ns + max(0, n - r0)
    return n - nw, nw


def decode_bytes_win(seq_lens, h_kv, h_q, sink, recent, group=32):
    """Algorithmic bytes of one decode with BF16 windows: the record (96 or
    72 B) per INT2 token and KV head, 512 B (bf16 K and V rows) per window
    token and KV head, bf16 query, fp32 output."""
    i2 = wt = 0
    for x in seq_lens:
        a, b = window_split(int(x), sink, recent)
        i2 += a
        wt += b
    B = len(seq_lens)
    return (i2 * h_kv * record_bytes(group) + wt * h_kv * 512 + B * h_q * D * 2 +
            B * h_q * D * 4)


# ------------------------------------------------------------------- ours

class Flusher:
    def __init__(self, dev):
        self.buf = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    def __call__(self):
        self.buf.fill_(1.0)


def setup_decode(name, seed, dev, variant, append_variant, batch=None):
    from paper_2608_02691_gb300 import optr, synth
    wl = synth.workload(name, seed)
    if batch:
        wl.B = batch
        wl.ctx = [wl.ctx[0]] * batch
    case = synth.build_case(wl, seed, device=dev)
    p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                case["h_q"], decode_variant=variant,
                                append_variant=append_variant)
    pool = optr.new_pool(p, case["num_pages"], device=dev)
    bt = case["block_table"].to(dev)
    cu = case["cu_ctx"]
    cl = cu.tolist()
    # prefill in chunks of whole sequences (bounded temporary memory): the
    # chunk's token rows are cu[b0]..cu[b1]; clamping the cumulative counts
    # to that window gives every other sequence zero new tokens.
    step = max(1, (1 << 21) // max(1, max(wl.ctx)))
    for b0 in range(0, case["B"], step):
        b1 = min(case["B"], b0 + step)
        if cl[b1] == cl[b0]:
            continue
        cu_sub = (cu.clamp(cl[b0], cl[b1]) - cl[b0]).to(torch.int32)
        optr.optr_kv_append(p, case["k_ctx"][cl[b0]:cl[b1]],
                            case["v_ctx"][cl[b0]:cl[b1]], cu_sub.to(dev),
                            case["pos0_ctx"].to(dev), bt, pool)
    torch.cuda.synchronize()
    return wl, case, p, pool, bt


def run_ours(args, rank, world, dev):
    from paper_2608_02691_gb300 import optr, synth
    hbm_peak, peak_src = peaks()
    flush = Flusher(dev)
    result = {}

    # ---------------- main step: decode8k (append 1 token/seq + decode)
    wl, case, p, pool, bt = setup_decode("decode8k", rank_seed(args.seed, rank),
                                         dev, args.variant, args.append_variant,
                                         args.batch)
    B, h_q, h_kv = case["B"], case["h_q"], case["h_kv"]
    seq = case["seq_lens"].to(dev)
    q = case["q"].to(dev)
    k_new, v_new = case["k_new"].to(dev), case["v_new"].to(dev)
    cu_new, pos0 = case["cu_new"].to(dev), case["pos0_new"].to(dev)
    out = torch.empty(B, h_q, D, dtype=torch.float32, device=dev)
    ws = optr.new_workspace(p, B, bt.shape[1], device=dev)
    stream = torch.cuda.current_stream()

    def step():
        # the cache write of the step's new tokens, then decode over the
        # updated cache (optr_kv_append + optr_decode_attention in one call)
        optr.optr_decode_step(p, q, k_new, v_new, cu_new, pos0, bt, seq, pool,
                              out, ws)

    step_bytes = (decode_bytes(case["seq_lens"].tolist(), h_kv, h_q) +
                  append_bytes(k_new.shape[0], h_kv))
    for _ in range(args.warmup):
        flush()
        step()
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0

    evs = [(torch.cuda.Event(enable_timing=True),
            torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    clocks = Clocks(torch.cuda.current_device()) if rank == 0 else None
    if clocks:
        clocks.start()
    barrier(world)
    torch.cuda.synchronize()
    for i in range(args.steps):
        flush()
        evs[i][0].record(stream)
        step()
        evs[i][1].record(stream)
    torch.cuda.synchronize()
    barrier(world)
    clk = clocks.stop() if clocks else None
    ms = float(np.mean([a.elapsed_time(b) for a, b in evs]))
    ms_max = allreduce_max(ms, world, dev)

    # stage breakdown (one step at a time, events recorded by the library)
    optr.optr_profile_enable(p, True)
    stages = {"append": [], "qrot": [], "partial": [], "combine": []}
    for _ in range(args.steps):
        flush()
        step()
        st = optr.optr_profile_last(p)
        for k2 in stages:
            stages[k2].append(st[k2])
    optr.optr_profile_enable(p, False)
    stage_ms = {k2: float(np.mean(v)) for k2, v in stages.items()}

    if args.no_e2e:
        e2e_ms, h2d, d2h, staged_ms = float("nan"), 0, 0, float("nan")
    else:
        e2e_ms, h2d, d2h, staged_ms = e2e_time(args, case, p, pool, bt, seq, cu_new,
                                               pos0, out, ws, flush, stream, world, dev)
    # roofline of the dominant kernel (split-K partial)
    part_bytes = decode_stream_bytes(case["seq_lens"].tolist(), h_kv)
    achieved = part_bytes / (stage_ms["partial"] * 1e-3) / 1e9
    variant_files = (["decode_tc.cu", "decode_common.cuh"]
                     if args.variant != 1 else ["decode.cu", "decode_common.cuh"])
    key = "partial_tensor" if args.variant != 1 else "partial_cuda_core"
    traffic = traffic_for(key, variant_files)
    roofline = {"bound": "hbm", "kernel": key, "achieved": round(achieved, 1),
                "peak": hbm_peak, "peak_source": peak_src, "unit": "GB/s",
                "frac": round(achieved / hbm_peak, 4),
                "frac_of_nominal_8000": round(achieved / 8000.0, 4),
                "traffic": traffic,
                "algorithmic_bytes_per_launch": part_bytes,
                "launch_ms": round(stage_ms["partial"], 5)}

    result["main"] = dict(ms=ms_max, bytes=step_bytes, stage_ms=stage_ms,
                          e2e_ms=e2e_ms, h2d=h2d, d2h=d2h, staged_ms=staged_ms,
                          roofline=roofline,
                          clocks=clk, case=case, pool=pool, p=p)
    return result


def e2e_time(args, case, p, pool, bt, seq, cu_new, pos0, out, ws, flush,
             stream, world, dev):
    """The step through the C ABI with HOST buffers: the query and the new
    K/V token of every sequence in pinned host memory, read in place by the
    step's kernels, and the output written by them to pinned host memory
    (the library's host-memory activations); every host-device transfer
    happens inside the timed region.  Also timed, for comparison: the same
    step on device buffers with explicit copy-engine transfers (one packed
    host-to-device copy, one device-to-host copy) around it."""
    from paper_2608_02691_gb300 import optr
    B, h_q = case["B"], case["h_q"]
    q_h = case["q"].cpu().contiguous().pin_memory()
    k_h = case["k_new"].cpu().contiguous().pin_memory()
    v_h = case["v_new"].cpu().contiguous().pin_memory()
    out_h = torch.empty(B, h_q, D, dtype=torch.float32).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in (q_h, k_h, v_h))
    d2h = out_h.numel() * out_h.element_size()

    def host_step():
        optr.optr_decode_step(p, q_h, k_h, v_h, cu_new, pos0, bt, seq, pool,
                              out_h, ws)

    # the copy-engine form: inputs packed in one pinned buffer
    parts = [q_h, k_h, v_h]
    sizes = [t.numel() * 2 for t in parts]
    in_h = torch.empty(h2d, dtype=torch.uint8).pin_memory()
    off = 0
    for t, n in zip(parts, sizes):
        in_h[off:off + n].copy_(t.view(torch.uint8).reshape(-1))
        off += n
    in_d = torch.empty(h2d, dtype=torch.uint8, device=dev)
    views, off = [], 0
    for t, n in zip(parts, sizes):
        views.append(in_d[off:off + n].view(torch.bfloat16).view(t.shape))
        off += n
    q_d, k_d, v_d = views
    out_c = torch.empty_like(out_h).pin_memory()

    def staged_step():
        in_d.copy_(in_h, non_blocking=True)
        optr.optr_decode_step(p, q_d, k_d, v_d, cu_new, pos0, bt, seq, pool,
                              out, ws)
        out_c.copy_(out, non_blocking=True)

    def timed(fn):
        for _ in range(args.warmup):
            flush()
            fn()
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True),
               torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        for i in range(args.steps):
            flush()
            ev[i][0].record(stream)
            fn()
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        ms = float(np.mean([a.elapsed_time(b) for a, b in ev]))
        return allreduce_max(ms, world, dev)

    e2e_ms = timed(host_step)
    staged_ms = timed(staged_step)
    # both forms deliver the same output
    assert torch.equal(out_h, out_c), "host-buffer step differs from the staged step"
    return e2e_ms, h2d, d2h, staged_ms


def extra_workloads(args, dev):
    """Prefill append throughput and the other decode workloads."""
    from paper_2608_02691_gb300 import optr, synth
    hbm_peak, _ = peaks()
    flush = Flusher(dev)
    res = {}
    # prefill append: 4 x 32768 tokens, G = 32 and the paper's G = 128, both
    # on the tcgen05 cache write
    for key, group in (("prefill_append", 32), ("prefill_append_g128", 128)):
        wl = synth.workload("prefill", args.seed)
        case = synth.build_case(wl, args.seed, device=dev)
        p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                    case["h_q"], append_variant=args.append_variant,
                                    group=group)
        pool = optr.new_pool(p, case["num_pages"], device=dev)
        bt = case["block_table"].to(dev)
        k, v = case["k_new"].to(dev), case["v_new"].to(dev)
        cu, pos0 = case["cu_new"].to(dev), case["pos0_new"].to(dev)
        for _ in range(3):
            optr.optr_kv_append(p, k, v, cu, pos0, bt, pool)
        optr.optr_profile_enable(p, True)
        t = []
        for _ in range(max(5, args.steps // 4)):
            flush()
            optr.optr_kv_append(p, k, v, cu, pos0, bt, pool)
            t.append(optr.optr_profile_last(p)["append"])
        optr.optr_profile_enable(p, False)
        ms = float(np.mean(t))
        n_tok = k.shape[0]
        nb = append_bytes(n_tok, case["h_kv"], group)
        res[key] = {
            "tokens": n_tok, "group": group, "ms": round(ms, 4),
            "tokens_per_s": round(n_tok / (ms * 1e-3), 1),
            "gbs": round(nb / (ms * 1e-3) / 1e9, 1),
            "frac": round(nb / (ms * 1e-3) / 1e9 / hbm_peak, 4)}
        del pool, k, v, case
        torch.cuda.empty_cache()

    res["decode8k_windows"] = windows_step(args, dev, flush, hbm_peak)
    torch.cuda.empty_cache()
    res["decode8k_paper_defaults"] = windows_step(args, dev, flush, hbm_peak,
                                                  group=128, clip_k=0.96,
                                                  clip_v=0.92)
    torch.cuda.empty_cache()
    # the compact G = 128 record (72 B per token and KV head) without windows
    res["decode8k_g128"] = windows_step(args, dev, flush, hbm_peak, sink=0,
                                        recent=0, group=128, clip_k=0.96,
                                        clip_v=0.92)
    torch.cuda.empty_cache()

    for name in ("long128k", "ragged"):
        wl, case, p, pool, bt = setup_decode(name, args.seed, dev, args.variant,
                                             args.append_variant)
        seq = case["seq_lens"].to(dev)
        q = case["q"].to(dev)
        out = torch.empty(case["B"], case["h_q"], D, device=dev)
        ws = optr.new_workspace(p, case["B"], bt.shape[1], device=dev)
        if case["k_new"].shape[0]:
            optr.optr_kv_append(p, case["k_new"].to(dev), case["v_new"].to(dev),
                                case["cu_new"].to(dev), case["pos0_new"].to(dev),
                                bt, pool)
        else:
            seq = case["seq_lens_ctx"].to(dev)
        for _ in range(3):
            optr.optr_decode_attention(p, q, bt, seq, pool, out, ws)
        optr.optr_profile_enable(p, True)
        st = []
        for _ in range(max(5, args.steps // 4)):
            flush()
            optr.optr_decode_attention(p, q, bt, seq, pool, out, ws)
            st.append(optr.optr_profile_last(p))
        optr.optr_profile_enable(p, False)
        lens = seq.cpu().tolist()
        tot = sum(np.mean([s[k2] for s in st]) for k2 in ("qrot", "partial", "combine"))
        part = float(np.mean([s["partial"] for s in st]))
        nb = decode_bytes(lens, case["h_kv"], case["h_q"])
        sb = decode_stream_bytes(lens, case["h_kv"])
        res[name] = {"decode_ms": round(tot, 4), "gbs": round(nb / (tot * 1e-3) / 1e9, 1),
                     "partial_ms": round(part, 4),
                     "partial_gbs": round(sb / (part * 1e-3) / 1e9, 1),
                     "partial_frac": round(sb / (part * 1e-3) / 1e9 / hbm_peak, 4)}
        del pool, case
        torch.cuda.empty_cache()
    res["calibration"] = calibration_workload(args, dev)
    return res


def calib_flops(T, nt, g, dm, steps, every, held=True):
    """Float64 FLOPs of optr_calibrate_head counted from its GEMM shapes
    (2 M N K each): per Adam step the forward and backward GEMMs of the
    objective, the rotation's exp (18 Horner products) and the Frechet
    derivative (3 per Horner step); squarings, whose count the device
    decides, are left out, so this is a lower bound."""
    d = 128
    key_f = 4 * T * d * d + 4 * g * nt * T * d + 2 * g * nt * d * dm
    key_b = 2 * g * nt * dm * d + 4 * g * nt * T * d + 6 * T * d * d
    val_f = 4 * T * d * d + 2 * g * nt * T * d + 2 * g * nt * d * dm
    val_b = 2 * g * nt * dm * d + 2 * g * nt * T * d + 6 * T * d * d
    rot = 19 * 2 * d ** 3
    grad = (3 * 18 + 1) * 2 * d ** 3
    n_sel = steps // every + (1 if steps % every else 0) + 1
    setup = 2 * (2 * g * nt * T * d) + 2 * key_f
    return (setup + steps * (key_f + key_b + val_f + val_b + 2 * (rot + grad))
            + n_sel * (key_f + val_f) + 2 * (steps + 1) * rot)


def calibration_workload(args, dev):
    """One KV head's calibration at the paper's scale (Sec. 5 and the
    appendix: ~2.7k-token traces, the objective over the final 64 query
    positions, 80 Adam steps, selection every 20 steps): a 2048-token
    synthetic trace and a held-out one of the same size, 4 query heads,
    d_model 4096 (Qwen3-8B), G = 128, clips 0.96 / 0.92, windows 64 / 256.
    The oracle is timed on one forward + backward of L_K at the same size."""
    from paper_2608_02691_gb300 import optr, synth
    T, nt, g, dm, steps, every = 2048, 64, 4, 4096, 80, 20
    tr = synth.calib_trace(args.seed, T, nt, g, dm)
    ho = synth.calib_trace(args.seed + 1, T, nt, g, dm)
    cfg = optr.calib_config(g, dm, T, nt, T, nt, steps=steps, select_every=every,
                            group=128, sink=64, recent=256, lr=0.02, lam=1.0,
                            clip_k=0.96, clip_v=0.92)
    q, K, V, W, tp = [x.to(dev) for x in tr]
    hd = tuple(x.to(dev) for x in (ho[0], ho[1], ho[2], ho[4]))
    optr.optr_calibrate_head(cfg, q, K, V, tp, W, held=hd)  # warm-up
    t = []
    for _ in range(2):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        optr.optr_calibrate_head(cfg, q, K, V, tp, W, held=hd)
        e1.record()
        torch.cuda.synchronize()
        t.append(e0.elapsed_time(e1) * 1e-3)
    sec = float(np.mean(t))
    flops = calib_flops(T, nt, g, dm, steps, every)
    gf = flops / sec / 1e9
    res = {"trace_tokens": T, "query_positions": nt, "query_heads": g,
           "d_model": dm, "steps": steps, "s_per_head": round(sec, 4),
           "qwen3_8b_all_heads_s": round(sec * 36 * 8, 1),
           "roofline": {"bound": "alu", "unit": "GFLOP/s", "dtype": "f64",
                        "achieved_lower_bound": round(gf, 1), "peak": 1250.0,
                        "peak_source": "nominal GB300 FP64 (not measured)",
                        "frac": round(gf / 1250.0, 4)}}
    if not args.no_cpu:
        import time
        from oracle import calibration as cal
        qc, Kc, Vc, Wc, tc = tr
        mu = Kc.mean(0)
        A = torch.zeros(128, 128, dtype=torch.float64, requires_grad=True)
        t0 = time.perf_counter()
        L = cal.key_loss(qc, Kc, Vc, mu, cal.rotation(cal.hadamard(128), A), Wc,
                         tc.long(), 1.0, 0.96, 128, 64, 256)
        torch.autograd.grad(L, A)
        st = time.perf_counter() - t0
        res["oracle"] = {"s_per_key_step": round(st, 3),
                         "cores": torch.get_num_threads(),
                         "s_per_head_est": round(st * 2 * steps, 1),
                         "sample": "one L_K forward + backward at the same size; "
                                   "per-head estimate = 160 such steps"}
    return res


def windows_step(args, dev, flush, hbm_peak, sink=64, recent=256, group=32,
                 clip_k=1.0, clip_v=1.0):
    """The decode8k step with the paper's BF16 windows (64 sink, 256 recent
    tokens; Sec. 5), optionally with its G = 128 and clip ratios:
    optr_decode_step_win, L2 flushed before every step.  sink = recent = 0:
    the same step without windows (optr_decode_step)."""
    from paper_2608_02691_gb300 import optr, synth
    wl = synth.workload("decode8k", args.seed)
    case = synth.build_case(wl, args.seed, device=dev)
    p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                case["h_q"], decode_variant=args.variant,
                                append_variant=args.append_variant, sink=sink,
                                recent=recent, group=group, clip_k=clip_k,
                                clip_v=clip_v)
    B, h_q, h_kv = case["B"], case["h_q"], case["h_kv"]
    pool = optr.new_pool(p, case["num_pages"], device=dev)
    windows = sink > 0 or recent > 0
    bt = case["block_table"].to(dev)
    if windows:
        win = optr.new_windows(p, B, device=dev)
        slot = torch.arange(B, dtype=torch.int32, device=dev)
        optr.optr_kv_append_win(p, case["k_ctx"], case["v_ctx"],
                                case["cu_ctx"].to(dev), case["pos0_ctx"].to(dev),
                                bt, pool, win, slot)
    else:
        optr.optr_kv_append(p, case["k_ctx"], case["v_ctx"], case["cu_ctx"].to(dev),
                            case["pos0_ctx"].to(dev), bt, pool)
    seq = case["seq_lens"].to(dev)
    q = case["q"].to(dev)
    k_new, v_new = case["k_new"].to(dev), case["v_new"].to(dev)
    cu_new, pos0 = case["cu_new"].to(dev), case["pos0_new"].to(dev)
    out = torch.empty(B, h_q, D, dtype=torch.float32, device=dev)
    ws = optr.new_workspace(p, B, bt.shape[1], device=dev)
    stream = torch.cuda.current_stream()

    def step():
        if windows:
            optr.optr_decode_step_win(p, q, k_new, v_new, cu_new, pos0, bt, seq,
                                      pool, win, slot, out, ws)
        else:
            optr.optr_decode_step(p, q, k_new, v_new, cu_new, pos0, bt, seq,
                                  pool, out, ws)

    for _ in range(3):
        flush()
        step()
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    n = max(5, args.steps // 2)
    evs = [(torch.cuda.Event(enable_timing=True),
            torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    for i in range(n):
        flush()
        evs[i][0].record(stream)
        step()
        evs[i][1].record(stream)
    torch.cuda.synchronize()
    ms = float(np.mean([a.elapsed_time(b) for a, b in evs]))
    optr.optr_profile_enable(p, True)
    part = []
    for _ in range(n):
        flush()
        step()
        part.append(optr.optr_profile_last(p)["partial"])
    optr.optr_profile_enable(p, False)
    lens = case["seq_lens"].tolist()
    n_new = k_new.shape[0]
    nb = (decode_bytes_win(lens, h_kv, h_q, sink, recent, group) +
          append_bytes(n_new, h_kv, group) +
          (n_new * h_kv * 512 if windows else 0))  # + window copies
    i2 = sum(window_split(x, sink, recent)[0] for x in lens)
    wt = sum(window_split(x, sink, recent)[1] for x in lens)
    pb = i2 * h_kv * record_bytes(group) + wt * h_kv * 512  # what the partial kernel streams
    pm = float(np.mean(part))
    return {"sink": sink, "recent": recent, "group": group,
            "clip_k": clip_k, "clip_v": clip_v, "step_ms": round(ms, 4),
            "bytes_per_step": nb, "gbs": round(nb / (ms * 1e-3) / 1e9, 1),
            "partial_ms": round(pm, 4),
            "partial_gbs": round(pb / (pm * 1e-3) / 1e9, 1),
            "partial_frac": round(pb / (pm * 1e-3) / 1e9 / hbm_peak, 4)}


# ---------------------------------------------------------- CPU baseline

def oracle_sample(case, n_seqs, threads):
    """The oracle, as it stands, on the first n_seqs sequences of a decode
    workload: its own cache write of their context (untimed set-up), then a
    step() closure = oracle append of their new token + oracle decode of all
    their query heads over the full context.  Inputs come from the seeded
    generator only.  Returns (step, bytes_per_step, description)."""
    from oracle import oracle
    from paper_2608_02691_gb300 import synth
    oracle.build()
    oracle.set_threads(threads)
    B = n_seqs
    cu = case["cu_ctx"][:B + 1]
    n_ctx = int(cu[-1])
    h_kv, h_q = case["h_kv"], case["h_q"]
    bt = case["block_table"][:B].numpy()
    used = np.unique(bt[bt >= 0])
    remap = np.full(case["num_pages"], -1, np.int64)
    remap[used] = np.arange(used.size)
    bt = np.where(bt >= 0, remap[np.maximum(bt, 0)], -1).astype(np.int32)
    pool = np.zeros((used.size, h_kv, CHUNK), np.uint8)
    R = (case["R_k"].numpy(), case["R_v"].numpy(), case["mu"].numpy())
    oracle.kv_append(synth.bf16_bits(case["k_ctx"][:n_ctx]),
                     synth.bf16_bits(case["v_ctx"][:n_ctx]), cu.numpy(),
                     case["pos0_ctx"][:B].numpy(), bt, pool, *R)
    n_new = int(case["cu_new"][B])
    kb = synth.bf16_bits(case["k_new"][:n_new])
    vb = synth.bf16_bits(case["v_new"][:n_new])
    qb = synth.bf16_bits(case["q"][:B])
    cu_new = case["cu_new"][:B + 1].numpy()
    pos0 = case["pos0_new"][:B].numpy()
    lens = case["seq_lens"][:B].numpy()

    def step():
        oracle.kv_append(kb, vb, cu_new, pos0, bt, pool, *R)
        oracle.decode_attention(qb, bt, lens, pool, R[0], R[1], h_kv)

    nb = decode_bytes(lens.tolist(), h_kv, h_q) + append_bytes(n_new, h_kv)
    desc = (f"{B} of {case['B']} sequences of the batch-{case['B']} x "
            f"{int(lens[0])}-token decode step (append 1 token + decode, all "
            f"{h_kv} KV heads / {h_q} query heads)")
    return step, nb, desc


def cpu_baseline(case, n_seqs, threads, reps=2):
    step, nb, desc = oracle_sample(case, n_seqs, threads)
    step()
    t0 = time.perf_counter()
    for _ in range(reps):
        step()
    dt = (time.perf_counter() - t0) / reps
    return {"value": round(nb / dt / 1e9, 4), "unit": "GB/s", "cores": threads,
            "kind": "oracle", "seconds_per_step": round(dt, 3), "sample": desc}


# ------------------------------------------------------------- reference

def run_reference(args, rank, world):
    """The oracle as the reference arm, on the same workload, metric and
    unit: each step is the oracle's decode step on a bounded sample."""
    if rank != 0:
        return None
    from paper_2608_02691_gb300 import synth
    threads = os.cpu_count() or 1
    case = synth.build_case(synth.workload("decode8k", args.seed), args.seed)
    step, nb, desc = oracle_sample(case, args.ref_seqs, threads)
    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = (time.perf_counter() - t0) / args.steps
    v = nb / dt / 1e9
    return {"impl": "reference", "metric": METRIC, "value": round(v, 4),
            "unit": "GB/s", "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(dt * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD_DESC, "sample_sequences": args.ref_seqs},
            "cpu_baseline": {"value": round(v, 4), "unit": "GB/s",
                             "cores": threads, "kind": "oracle", "sample": desc},
            "e2e": {"value": round(v, 4), "unit": "GB/s",
                    "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


WORKLOAD_DESC = ("decode8k: batch 16 x context 8192 (+1 appended token per "
                 "sequence), 32 q / 8 kv heads, head_dim 128, page 16, "
                 "shuffled pages, Student-t(4) K/V")
METRIC = "decode-attention HBM GB/s (decode step: append 1 token/seq + decode)"


# ------------------------------------------------------------- dist glue

def barrier(world):
    if world > 1:
        torch.distributed.barrier()


def rank_seed(seed, rank):
    """Each rank decodes its own independent batch (weak scaling: the
    sequences of a decode batch are independent problems, so ranks share no
    data and run no data-path collective)."""
    return seed + 1009 * rank


def job_value(bytes_per_rank, ms_max, world):
    """Whole-job GB/s: the bytes of all ranks over the slowest rank's time."""
    return bytes_per_rank * world / (ms_max * 1e-3) / 1e9


def allreduce_max(x, world, dev):
    if world <= 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--variant", type=int, default=0)
    ap.add_argument("--append-variant", type=int, default=0)
    ap.add_argument("--ref-seqs", type=int, default=4)
    ap.add_argument("--cpu-seqs", type=int, default=16)
    ap.add_argument("--no-extra", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--batch", type=int, default=0,
                    help="override the decode8k batch (profiling cases)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if world > 1:
            os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        line = run_reference(args, rank, world)
        if line is not None:
            print(json.dumps(line), flush=True)
        return

    if world > 1:
        torch.distributed.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import __graft_entry__
    __graft_entry__.build()

    res = run_ours(args, rank, world, dev)
    m = res["main"]
    # the other workloads only at N = 1 (a multi-GPU run holds every GPU)
    extra = (extra_workloads(args, dev)
             if (rank == 0 and world == 1 and not args.no_extra) else None)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        case_cpu = {k: (v.cpu() if torch.is_tensor(v) else v)
                    for k, v in m["case"].items()}
        del m["pool"], m["case"]
        cpu = cpu_baseline(case_cpu, args.cpu_seqs, os.cpu_count() or 1)
        # the same oracle on one host core, on one sequence of the batch
        one = cpu_baseline(case_cpu, 1, 1)
        cpu["single_thread"] = {k: one[k] for k in ("value", "unit", "cores",
                                                    "seconds_per_step", "sample")}
    if rank == 0:
        value = job_value(m["bytes"], m["ms"], world)
        e2e = (None if not np.isfinite(m["e2e_ms"]) else
               job_value(m["bytes"], m["e2e_ms"], world))
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": "GB/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(m["ms"], 5), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int2+fp16 meta, f32 math",
            "data": "synthetic",
            "config": {"workload": WORKLOAD_DESC,
                       "bytes_per_step": m["bytes"], "l2": "flushed (512 MiB write) "
                       "before every timed step; step timed alone with CUDA events",
                       "decode_variant": args.variant, "append_variant": args.append_variant},
            # optr_decode_step: fused cache write + query rotation, partial,
            # combine (4 launches when a CUDA-core variant is selected)
            "gpu_launches": (3 if args.variant != 1 and args.append_variant != 1
                             else 4) * args.steps,
            "stage_ms": {k: round(v, 5) for k, v in m["stage_ms"].items()},
            "roofline": m["roofline"],
            "e2e": None if e2e is None else {
                "value": round(e2e, 2), "unit": "GB/s",
                "h2d_bytes_per_step": m["h2d"], "d2h_bytes_per_step": m["d2h"],
                "ms_per_step": round(m["e2e_ms"], 5),
                "mode": "optr_decode_step with q, k_new, v_new and out in pinned "
                        "host memory: the step's kernels read the inputs and write "
                        "the output over NVLink-C2C inside the timed region",
                "staged_copy_engine": {
                    "value": round(job_value(m["bytes"], m["staged_ms"], world), 2),
                    "ms_per_step": round(m["staged_ms"], 5),
                    "mode": "device buffers, one packed host-to-device and one "
                            "device-to-host cudaMemcpyAsync around the step"}},
            "clocks": m["clocks"],
            "cpu_baseline": cpu,
            "workloads": extra,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
