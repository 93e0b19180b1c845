"""GPU parity: the CUDA library against the fp64 CPU oracle, element by
element, on seeded inputs of the five workloads at sizes the oracle finishes
in seconds (several pages per sequence, ragged tails, shuffled pages), plus
edge cases.  Every call goes through the C ABI (liboptr.so)."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_02691_gb300 import optr, synth

import parity_helpers as ph

pytestmark = pytest.mark.gpu

VARIANTS = [optr.OPTR_VARIANT_CUDA_CORE]
APPEND_VARIANTS = [optr.OPTR_VARIANT_CUDA_CORE]
CASES = [("tiny", 1.0), ("decode8k", 1 / 16), ("long128k", 1 / 32),
         ("prefill", 1 / 128), ("ragged", 1 / 32)]


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


def _case(name, scale, seed=0):
    key = (name, scale, seed)
    if key not in _cache:
        c = synth.build_case(synth.workload(name, seed, scale), seed)
        pool, u_ctx, u_new = ph.oracle_case(c)
        _cache[key] = (c, pool, u_ctx, u_new)
    return _cache[key]


@pytest.mark.parametrize("name,scale", CASES)
@pytest.mark.parametrize("avar", APPEND_VARIANTS)
def test_append_matches_oracle(name, scale, avar):
    c, pool_ref, u_ctx, u_new = _case(name, scale)
    p, pool, _ = ph.gpu_case(c, append_variant=avar)
    assert optr.optr_device_error(p) == 0
    pg = pool.cpu().numpy()
    for k, cu, pos0, u in (("ctx", c["cu_ctx"], c["pos0_ctx"], u_ctx),
                           ("new", c["cu_new"], c["pos0_new"], u_new)):
        if u is None:
            continue
        pages, slots = ph.token_slots(cu, pos0, c["block_table"])
        st = ph.compare_append(pg, pool_ref, u, pages, slots)
        print(f"{name} {k}: {st}")


@pytest.mark.parametrize("name,scale", CASES)
@pytest.mark.parametrize("variant", VARIANTS)
def test_decode_matches_oracle(name, scale, variant):
    c, pool_ref, _, _ = _case(name, scale)
    p, pool, out = ph.gpu_case(c, variant=variant)
    assert optr.optr_device_error(p) == 0
    got = out.cpu().double().numpy()
    # decode error alone: oracle decode over the GPU-written cache
    ref = ph.oracle_decode(c, pool.cpu().numpy())
    r1 = ph.assert_decode_close(got, ref, f"{name} decode")
    # end to end: oracle append + oracle decode
    ref2 = ph.oracle_decode(c, pool_ref)
    r2 = ph.assert_decode_close(got, ref2, f"{name} end-to-end")
    print(f"{name} variant {variant}: err/rms decode {r1:.2e} e2e {r2:.2e}")


@pytest.mark.parametrize("variant", VARIANTS)
def test_unused_slots_never_read(variant):
    """Slots past seq_len hold NaN metadata (pool pre-filled with 0xFF): the
    output stays finite and equal to the oracle's."""
    c, _, _, _ = _case("ragged", 1 / 32)
    p, pool, out = ph.gpu_case(c, variant=variant, poison=True)
    got = out.cpu().double().numpy()
    ref = ph.oracle_decode(c, pool.cpu().numpy())
    ph.assert_decode_close(got, ref, "poisoned")


@pytest.mark.parametrize("variant", VARIANTS)
def test_sequence_length_edges(variant):
    """seq_len 0 (zeros), 1, 15, 16, 17, 31, 33 over one prefilled cache."""
    c, _, _, _ = _case("decode8k", 1 / 16)
    p, pool, _ = ph.gpu_case(c, variant=variant)
    lens = torch.tensor([0, 1, 15, 16, 17, 31, 33, 2, 3, 100, 257, 511, 512,
                         513, 64, 48], dtype=torch.int32)
    dev = "cuda"
    out = torch.full((c["B"], c["h_q"], 128), 7.0, device=dev)
    ws = optr.new_workspace(p, c["B"], c["block_table"].shape[1])
    optr.optr_decode_attention(p, c["q"].to(dev), c["block_table"].to(dev),
                               lens.to(dev), pool, out, ws)
    got = out.cpu().double().numpy()
    assert not got[0].any()
    ref = ph.oracle_decode(c, pool.cpu().numpy(), seq_lens=lens)
    ph.assert_decode_close(got, ref, "length edges")
    assert optr.optr_device_error(p) == 0


@pytest.mark.parametrize("variant", VARIANTS)
def test_split_invariance(variant):
    """The split-K cut points of a sequence depend on the whole batch; the
    result for one sequence must not (alone vs inside the batch)."""
    c, _, _, _ = _case("ragged", 1 / 32)
    p, pool, out = ph.gpu_case(c, variant=variant)
    dev = "cuda"
    bt = c["block_table"]
    for b in (0, 7, 127):
        o1 = torch.empty(1, c["h_q"], 128, device=dev)
        ws = optr.new_workspace(p, 1, bt.shape[1])
        optr.optr_decode_attention(p, c["q"][b:b + 1].to(dev),
                                   bt[b:b + 1].contiguous().to(dev),
                                   c["seq_lens"][b:b + 1].to(dev), pool, o1, ws)
        torch.cuda.synchronize()
        a, bb = o1[0].double().cpu(), out[b].double().cpu()
        rms = float(a.pow(2).mean().sqrt())
        assert float((a - bb).abs().max()) <= 1e-5 * rms


def test_needle_is_retrieved():
    """long-context workload: the planted key wins the softmax of its
    group's first query head, and the GPU output matches the oracle."""
    c, _, _, _ = _case("long128k", 1 / 16)
    p, pool, out = ph.gpu_case(c)
    pn = pool.cpu().numpy()
    for h, pos in enumerate(c["needle"].tolist()):
        j = 4 * h
        _, prob = oracle.decode_attention(
            synth.bf16_bits(c["q"]), c["block_table"].numpy(),
            c["seq_lens"].numpy(), pn, c["R_k"].numpy(), c["R_v"].numpy(),
            c["h_kv"], rows=[(0, j)], want_p=True)
        assert int(np.argmax(prob)) == pos
    ref = ph.oracle_decode(c, pn)
    ph.assert_decode_close(out.cpu().double().numpy(), ref, "needle")


def test_bad_tables_are_flagged_not_read():
    c, _, _, _ = _case("decode8k", 1 / 16)
    p, pool, _ = ph.gpu_case(c)
    dev = "cuda"
    bt = c["block_table"].clone()
    bt[3, 2] = c["num_pages"] + 5
    out = torch.empty(c["B"], c["h_q"], 128, device=dev)
    ws = optr.new_workspace(p, c["B"], bt.shape[1])
    optr.optr_decode_attention(p, c["q"].to(dev), bt.to(dev),
                               c["seq_lens"].to(dev), pool, out, ws)
    assert optr.optr_device_error(p) & 1
    # append at a position beyond the table
    pos0 = torch.full((c["B"],), bt.shape[1] * 16, dtype=torch.int32)
    optr.optr_kv_append(p, c["k_new"].to(dev), c["v_new"].to(dev),
                        c["cu_new"].to(dev), pos0.to(dev), bt.to(dev), pool)
    assert optr.optr_device_error(p) & 2
    lens = c["seq_lens"].clone()
    lens[0] = bt.shape[1] * 16 + 1
    optr.optr_decode_attention(p, c["q"].to(dev), c["block_table"].to(dev),
                               lens.to(dev), pool, out, ws)
    assert optr.optr_device_error(p) & 4
    assert optr.optr_device_error(p) == 0


def test_workspace_too_small_is_rejected():
    c, _, _, _ = _case("tiny", 1.0)
    p, pool, out = ph.gpu_case(c)
    ws = torch.empty(128, dtype=torch.uint8, device="cuda")
    with pytest.raises(optr.OptrError) as e:
        optr.optr_decode_attention(p, c["q"].cuda(), c["block_table"].cuda(),
                                   c["seq_lens"].cuda(), pool, out, ws)
    assert e.value.status == -4
