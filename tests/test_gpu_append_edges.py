"""Cache-write edge cases, both append variants against the oracle:

* clip ratios below 1 (the clamped quantizer, Sec. 3.1 clipping ratio c);
* more sequences than the kernels cache in shared memory (600 > 512), each
  a few tokens, so the tensor-core kernel resolves slots through global
  memory;
* 257 new tokens (one past the single-token kernel's limit) split over
  sequences whose first positions are not page-aligned, leaving the last
  128-token tile of the tensor-core kernel nearly empty;
* value groups of 32 channels that are constant (degenerate range: codes
  0, scale 0) next to ordinary ones.
"""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_02691_gb300 import optr, synth

import parity_helpers as ph

pytestmark = pytest.mark.gpu

H_KV, H_Q = 8, 32
APPEND_VARIANTS = [optr.OPTR_VARIANT_CUDA_CORE, optr.OPTR_VARIANT_TENSOR]


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02691_gb300 import build
    build.build()
    oracle.build()
    torch.cuda.set_device(0)


def _append_case(lens, first_pos, seed, degenerate=False):
    """New tokens of len(lens) sequences, sequence b's first token at cache
    position first_pos[b]; shuffled page table covering every position."""
    lens = [int(x) for x in lens]
    first_pos = [int(x) for x in first_pos]
    n_tok = sum(lens)
    k, v = synth.kv_tokens(n_tok, H_KV, "t4", seed, 3)
    R_k, R_v = synth.rotations(H_KV, seed)
    if degenerate:
        # every fourth token: value group 1 constant, with R_v = I
        v[::4, :, 32:64] = -0.75
        R_v = torch.eye(128).expand(H_KV, 128, 128).contiguous()
    mu = synth.key_mean(k)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    bt, num_pages = synth.page_tables([p + n for p, n in zip(first_pos, lens)],
                                      True, seed)
    return dict(k=k, v=v, R_k=R_k, R_v=R_v, mu=mu, cu=cu,
                pos0=np.array(first_pos, np.int32), bt=bt, num_pages=num_pages)


def _check(c, avar, clip_k=1.0, clip_v=1.0):
    bt = c["bt"]
    pool_ref = np.zeros((c["num_pages"], H_KV, 1536), np.uint8)
    u = oracle.kv_append(synth.bf16_bits(c["k"]), synth.bf16_bits(c["v"]),
                         c["cu"], c["pos0"], bt.numpy(), pool_ref,
                         c["R_k"].numpy(), c["R_v"].numpy(), c["mu"].numpy(),
                         clip_k=clip_k, clip_v=clip_v, want_u=True)
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], H_Q, clip_k=clip_k,
                                clip_v=clip_v, append_variant=avar)
    pool = optr.new_pool(p, c["num_pages"], device="cuda")
    optr.optr_kv_append(p, c["k"].cuda(), c["v"].cuda(),
                        torch.from_numpy(c["cu"]).cuda(),
                        torch.from_numpy(c["pos0"]).cuda(), bt.cuda(), pool)
    torch.cuda.synchronize()
    assert optr.optr_device_error(p) == 0
    pages, slots = ph.token_slots(c["cu"], c["pos0"], bt.numpy())
    return ph.compare_append(pool.cpu().numpy(), pool_ref, u, pages, slots)


@pytest.mark.parametrize("avar", APPEND_VARIANTS)
@pytest.mark.parametrize("clip_k,clip_v", [(0.9, 0.8), (0.5, 1.0)])
def test_clip_ratio_below_one(avar, clip_k, clip_v):
    g = np.random.default_rng(11)
    lens = g.integers(40, 400, size=6)
    first = g.integers(0, 40, size=6)
    st = _check(_append_case(lens, first, 21), avar, clip_k, clip_v)
    assert st["codes"] > 0


@pytest.mark.parametrize("avar", APPEND_VARIANTS)
def test_more_sequences_than_cached(avar):
    g = np.random.default_rng(12)
    lens = g.integers(1, 4, size=600)
    first = g.integers(0, 50, size=600)
    st = _check(_append_case(lens, first, 22), avar)
    assert st["codes"] == 2 * int(lens.sum()) * H_KV * 128


@pytest.mark.parametrize("avar", APPEND_VARIANTS)
def test_just_past_single_token_limit(avar):
    lens = [100, 100, 57]  # 257 tokens: the tensor-core kernel, 3 tiles
    first = [7, 16, 31]
    _check(_append_case(lens, first, 23), avar)


@pytest.mark.parametrize("avar", APPEND_VARIANTS)
def test_degenerate_groups(avar):
    lens = [300, 45]
    first = [3, 0]
    c = _append_case(lens, first, 24, degenerate=True)
    _check(c, avar)
    # the constant groups stored scale 0 and every code 0 (oracle pins the
    # same rule); checked here on the GPU pool through the oracle compare
    # above, and directly on one record:
    p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], H_Q, append_variant=avar)
    pool = optr.new_pool(p, c["num_pages"], device="cuda")
    optr.optr_kv_append(p, c["k"].cuda(), c["v"].cuda(),
                        torch.from_numpy(c["cu"]).cuda(),
                        torch.from_numpy(c["pos0"]).cuda(), c["bt"].cuda(), pool)
    torch.cuda.synchronize()
    pages, slots = ph.token_slots(c["cu"], c["pos0"], c["bt"].numpy())
    codes, scale, _ = ph.slot_codes(pool.cpu().numpy(), pages[:1], slots[:1], 1)
    assert scale[0, :, 1].max() == 0.0  # value group 1 of token 0
    assert codes[0, :, 32:64].max() == 0


def test_fp16_range_flag_on_tensor_variant():
    """The tensor-core cache write converts k and v to fp16: a key element
    of magnitude >= 65504 (bf16 70144 here) sets OPTR_DEVERR_FP16_RANGE and
    leaves only that token-head's key record unspecified; every other record
    still matches the oracle.  The CUDA-core variant takes the same input
    without the flag and matches the oracle on every record."""
    lens, first = [200, 100], [5, 0]
    c = _append_case(lens, first, 25)
    t_bad, h_bad = 17, 3
    c["k"][t_bad, h_bad, 5] = 70000.0  # bf16 rounds it to 70144
    assert float(c["k"][t_bad, h_bad, 5]) >= 65504.0
    bt = c["bt"]
    pool_ref = np.zeros((c["num_pages"], H_KV, 1536), np.uint8)
    u = oracle.kv_append(synth.bf16_bits(c["k"]), synth.bf16_bits(c["v"]),
                         c["cu"], c["pos0"], bt.numpy(), pool_ref,
                         c["R_k"].numpy(), c["R_v"].numpy(), c["mu"].numpy(),
                         want_u=True)
    pages, slots = ph.token_slots(c["cu"], c["pos0"], bt.numpy())
    for avar in APPEND_VARIANTS:
        p = optr.optr_params_create(c["R_k"], c["R_v"], c["mu"], H_Q,
                                    append_variant=avar)
        pool = optr.new_pool(p, c["num_pages"], device="cuda")
        optr.optr_kv_append(p, c["k"].cuda(), c["v"].cuda(),
                            torch.from_numpy(c["cu"]).cuda(),
                            torch.from_numpy(c["pos0"]).cuda(), bt.cuda(), pool)
        torch.cuda.synchronize()
        flags = optr.optr_device_error(p)
        got = pool.cpu().numpy()
        ref = pool_ref.copy()
        if avar == optr.OPTR_VARIANT_TENSOR:
            assert flags == optr.OPTR_DEVERR_FP16_RANGE
            # the flagged key record (codes and metadata) is unspecified
            pg, sl = pages[t_bad], slots[t_bad]
            for arr in (got, ref):
                arr[pg, h_bad, sl * 32:sl * 32 + 32] = 0
                arr[pg, h_bad, 1024 + sl * 16:1024 + sl * 16 + 16] = 0
        else:
            assert flags == 0
        ph.compare_append(got, ref, u, pages, slots)
