"""Parity at the full workload sizes, in the benchmark's launch configuration.

The whole batch of each decode workload (decode8k, long128k, ragged) is
decoded in one library call with the workspace and launch shape bench.py
times.  The oracle cannot decode every sequence of these batches in seconds,
so it writes the cache records of a few sampled sequences from its own
CPU-generated keys and values (same recipe: Student-t(4), the per-head key
offsets, the planted needle of long128k), those records are copied into the
GPU pool at the sampled sequences' physical pages, and the sampled outputs
are compared with the oracle's decode of the same records.  The other
sequences' pages hold a GPU-written cache of GPU-generated tokens, which
only keeps the batch at its full size; no expected value comes from them.

The prefill append (4 x 32768 tokens) is compared record by record on
sampled tokens; its inputs are generated on the CPU and fed to both sides.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_02691_gb300 import optr, synth
from parity_helpers import (OUT_TOL, compare_append, token_slots)

pytestmark = pytest.mark.gpu

DECODE_VARIANTS = [optr.OPTR_VARIANT_CUDA_CORE, optr.OPTR_VARIANT_TENSOR]
SAMPLES = {"decode8k": (0, 9, 15), "long128k": (0,), "ragged": (0, 63, 127)}
SEED = 0
_cache: dict = {}


def _gpu_full(name, group=32, clip_k=1.0, clip_v=1.0):
    """Full-size workload generated and appended on the GPU (as bench.py
    builds it), with the sampled sequences overwritten by oracle records.
    Returns (case, pool, per-sample (oracle output, b)).  group = 128 uses
    the compact record (1152 bytes per page and KV head) with the clips."""
    key = (name, group, clip_k, clip_v)
    if key in _cache:
        return _cache[key]
    dev = "cuda"
    wl = synth.workload(name, SEED)
    case = synth.build_case(wl, SEED, device=dev)
    p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                case["h_q"], group=group, clip_k=clip_k,
                                clip_v=clip_v)
    pool = optr.new_pool(p, case["num_pages"], device=dev)
    bt = case["block_table"].to(dev)
    optr.optr_kv_append(p, case["k_ctx"], case["v_ctx"],
                        case["cu_ctx"].to(dev), case["pos0_ctx"].to(dev), bt,
                        pool)
    if case["k_new"].shape[0]:
        optr.optr_kv_append(p, case["k_new"], case["v_new"],
                            case["cu_new"].to(dev), case["pos0_new"].to(dev),
                            bt, pool)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    del case["k_ctx"], case["v_ctx"]  # free the GPU-generated tokens

    h_kv, h_q = case["h_kv"], case["h_q"]
    R_k, R_v = case["R_k"].numpy(), case["R_v"].numpy()
    mu = case["mu"].numpy()
    q_cpu = case["q"].cpu()
    bt_cpu = case["block_table"]
    lens = case["seq_lens"].tolist()
    refs = []
    for i, b in enumerate(SAMPLES[name]):
        n = lens[b]
        k, v = synth.kv_tokens(n, h_kv, wl.dist, SEED, 100 + i, "cpu")
        if wl.needle and b == 0:
            synth.plant_needles(k, [0, n], case["mu"], q_cpu, SEED)
        npg = (n + 15) // 16
        obt = np.arange(npg, dtype=np.int32)[None]
        opool = np.zeros((npg, h_kv, oracle.chunk_bytes(group)), np.uint8)
        oracle.kv_append(synth.bf16_bits(k), synth.bf16_bits(v),
                         np.array([0, n], np.int32), np.zeros(1, np.int32),
                         obt, opool, R_k, R_v, mu, clip_k=clip_k,
                         clip_v=clip_v, group=group)
        ref = oracle.decode_attention(synth.bf16_bits(q_cpu[b:b + 1]), obt,
                                      np.array([n], np.int32), opool, R_k, R_v,
                                      h_kv)[0]
        phys = bt_cpu[b, :npg].to(torch.int64).to(dev)
        pool.index_copy_(0, phys, torch.from_numpy(opool).to(dev))
        refs.append((b, ref))
    torch.cuda.synchronize()
    _cache[key] = (case, pool, refs)
    return _cache[key]


@pytest.mark.parametrize("variant", DECODE_VARIANTS)
@pytest.mark.parametrize("name", list(SAMPLES))
def test_full_size_decode(name, variant):
    case, pool, refs = _gpu_full(name)
    dev = "cuda"
    p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                case["h_q"], decode_variant=variant)
    bt = case["block_table"].to(dev)
    out = torch.full((case["B"], case["h_q"], 128), 7.0, dtype=torch.float32,
                     device=dev)
    ws = optr.new_workspace(p, case["B"], bt.shape[1], device=dev)
    optr.optr_decode_attention(p, case["q"], bt, case["seq_lens"].to(dev),
                               pool, out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    got = out.cpu().double().numpy()
    assert np.all(np.isfinite(got))
    for b, ref in refs:
        rms = float(np.sqrt(np.mean(ref ** 2)))
        err = float(np.abs(got[b] - ref).max())
        print(f"{name} variant {variant} seq {b}: err/rms {err / rms:.2e}")
        assert err <= OUT_TOL * rms, (name, variant, b, err / rms)


@pytest.mark.parametrize("variant", DECODE_VARIANTS)
def test_full_size_decode_compact_g128(variant):
    """decode8k at full size with the paper's quantizer settings (G = 128,
    clips 0.96 / 0.92) in the compact record: 72 B per token and KV head."""
    case, pool, refs = _gpu_full("decode8k", 128, 0.96, 0.92)
    assert pool.shape[-1] == 1152
    dev = "cuda"
    p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                case["h_q"], decode_variant=variant, group=128,
                                clip_k=0.96, clip_v=0.92)
    bt = case["block_table"].to(dev)
    out = torch.full((case["B"], case["h_q"], 128), 7.0, dtype=torch.float32,
                     device=dev)
    ws = optr.new_workspace(p, case["B"], bt.shape[1], device=dev)
    optr.optr_decode_attention(p, case["q"], bt, case["seq_lens"].to(dev),
                               pool, out, ws)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    got = out.cpu().double().numpy()
    assert np.all(np.isfinite(got))
    for b, ref in refs:
        rms = float(np.sqrt(np.mean(ref ** 2)))
        err = float(np.abs(got[b] - ref).max())
        print(f"decode8k G=128 variant {variant} seq {b}: err/rms {err / rms:.2e}")
        assert err <= OUT_TOL * rms, (variant, b, err / rms)


@pytest.mark.parametrize("append_variant",
                         [optr.OPTR_VARIANT_CUDA_CORE, optr.OPTR_VARIANT_TENSOR])
def test_full_size_prefill_append(append_variant):
    wl = synth.workload("prefill", SEED)
    case = synth.build_case(wl, SEED, device="cpu")
    dev = "cuda"
    p = optr.optr_params_create(case["R_k"], case["R_v"], case["mu"],
                                case["h_q"], append_variant=append_variant)
    pool = optr.new_pool(p, case["num_pages"], device=dev)
    bt = case["block_table"]
    optr.optr_kv_append(p, case["k_new"].to(dev), case["v_new"].to(dev),
                        case["cu_new"].to(dev), case["pos0_new"].to(dev),
                        bt.to(dev), pool)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    gpu_pool = pool.cpu().numpy()

    # sampled tokens, each appended by the oracle as a one-token "sequence"
    n_tok = case["k_new"].shape[0]
    g = torch.Generator().manual_seed(5)
    sel = torch.randperm(n_tok, generator=g)[:4096].sort().values.numpy()
    cu = case["cu_new"].numpy()
    seq_of = np.searchsorted(cu, sel, side="right") - 1
    pos = case["pos0_new"].numpy()[seq_of] + sel - cu[seq_of]
    obt = bt.numpy()[seq_of]
    ocu = np.arange(len(sel) + 1, dtype=np.int32)
    opool = np.zeros_like(gpu_pool)
    u = oracle.kv_append(synth.bf16_bits(case["k_new"][sel]),
                         synth.bf16_bits(case["v_new"][sel]), ocu,
                         pos.astype(np.int32), obt, opool,
                         case["R_k"].numpy(), case["R_v"].numpy(),
                         case["mu"].numpy(), want_u=True)
    pages, slots = token_slots(ocu, pos.astype(np.int32), obt)
    st = compare_append(gpu_pool, opool, u, pages, slots)
    print(f"prefill append variant {append_variant}: {st['codes']} codes, "
          f"{st['tie_band']} in the tie band, {st['mismatch_in_band']} differ")
