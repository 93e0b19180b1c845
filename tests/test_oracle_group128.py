"""Pins of the oracle's G = 128 quantizer (Sec. 3.1: Q2 with group size G;
Sec. 5 and the default-settings table: G = 128, clipping ratios 0.96 for
keys and 0.92 for values).  With G = 128 one (scale, min) pair covers all
128 rotated channels; the stored layout keeps one pair per 32-channel
block, so the pair is repeated in its four blocks.
"""
import numpy as np
import pytest
import torch

from paper_2608_02691_gb300 import synth

D = 128
EYE = np.eye(D, dtype=np.float32)


def _f16(bits):
    return float(np.array([bits], np.uint16).view(np.float16)[0])


def test_hand_worked_128_group(oracle_mod):
    """Block 0 holds 0, 1, 2, 3 repeated, blocks 1-3 hold 0, 3, 6, 9
    repeated: the 128-group spans [0, 9], scale 3, min 0, so block 0's
    values map to u = z / 3 = 0, 1/3, 2/3, 1 -> codes 0, 0, 1, 1 and the
    other blocks' to u = 0, 1, 2, 3 -> codes 0, 1, 2, 3 (with G = 32
    block 0 would keep codes 0, 1, 2, 3 at scale 1)."""
    base = np.tile(np.arange(4.0), 8)
    z = np.concatenate([base, 3 * base, 3 * base, 3 * base])
    _, codes, s, m, _ = oracle_mod.rotate_quantize(z, EYE, group=128)
    np.testing.assert_array_equal(codes[:32], np.tile([0, 0, 1, 1], 8))
    np.testing.assert_array_equal(codes[32:], np.tile([0, 1, 2, 3], 24))
    assert all(_f16(x) == 3.0 for x in s) and all(_f16(x) == 0.0 for x in m)
    _, c32, s32, _, _ = oracle_mod.rotate_quantize(z, EYE, group=32)
    np.testing.assert_array_equal(c32[:32], base)
    assert _f16(s32[0]) == 1.0 and _f16(s32[1]) == 3.0


def test_128_group_equals_32_groups_when_blocks_share_the_range(oracle_mod):
    """If every 32-channel block has the same minimum and maximum, one
    128-group and four 32-groups quantize identically."""
    rng = np.random.default_rng(40)
    z = np.clip(rng.standard_normal(D), -2.4, 3.2)
    for blk in range(4):
        z[32 * blk] = -2.5
        z[32 * blk + 7] = 3.25
    a = oracle_mod.rotate_quantize(z, EYE, group=128)
    b = oracle_mod.rotate_quantize(z, EYE, group=32)
    for x, y in zip(a[1:4], b[1:4]):
        np.testing.assert_array_equal(x, y)


@pytest.mark.parametrize("clip", [1.0, 0.96, 0.92])
def test_128_group_error_bound(oracle_mod, clip):
    """|zhat - z| <= scale/2 (+ fp16 rounding of the metadata) inside the
    clipped range [c min, c max]; values outside it saturate at the ends."""
    rng = np.random.default_rng(41)
    for _ in range(20):
        z = rng.standard_t(4, D) * rng.uniform(0.1, 10)
        _, codes, s, m, _ = oracle_mod.rotate_quantize(z, EYE, clip, group=128)
        sc, mn = _f16(s[0]), _f16(m[0])
        zhat = codes * sc + mn
        lo, hi = clip * z.min(), clip * z.max()
        inside = (z >= lo) & (z <= hi)
        tol = sc / 2 + 3 * 2 ** -11 * (abs(mn) + 3 * sc)
        assert np.all(np.abs(zhat - z)[inside] <= tol)
        assert np.all(codes[z < lo] == 0) and np.all(codes[z > hi] == 3)
        assert len(set(s)) == 1 and len(set(m)) == 1


def test_paged_equals_dense_with_128_groups(oracle_mod):
    """Rotated-query form = inverse-rotation form with G = 128, the paper's
    clip ratios and windows (Appendix, rotated-query implementation)."""
    rng = np.random.default_rng(42)
    h_kv, h_q = 2, 8
    seq = [3, 40, 150]
    n = sum(seq)
    R_k, R_v = synth.rotations(h_kv, 3)
    k = torch.tensor(rng.standard_t(4, (n, h_kv, D)) +
                     np.where(rng.random((1, h_kv, D)) < 0.03, 8.0, 0.0),
                     dtype=torch.bfloat16)
    v = torch.tensor(rng.standard_t(4, (n, h_kv, D)), dtype=torch.bfloat16)
    q = torch.tensor(rng.standard_normal((len(seq), h_q, D)), dtype=torch.bfloat16)
    mu = synth.key_mean(k).numpy()
    bt, num_pages = synth.page_tables(seq, True, 3)
    cu = np.concatenate([[0], np.cumsum(seq)]).astype(np.int32)
    pos0 = np.zeros(len(seq), np.int32)
    pool = np.zeros((num_pages, h_kv, oracle_mod.chunk_bytes(128)), np.uint8)
    kb, vb = synth.bf16_bits(k), synth.bf16_bits(v)
    oracle_mod.kv_append(kb, vb, cu, pos0, bt.numpy(), pool, R_k.numpy(),
                         R_v.numpy(), mu, clip_k=0.96, clip_v=0.92, group=128)
    sink, recent = 16, 32
    win = oracle_mod.new_windows(len(seq), h_kv, sink, recent)
    slots = np.arange(len(seq), dtype=np.int32)
    oracle_mod.window_write(kb, vb, cu, pos0, win, slots, sink, recent)
    out = oracle_mod.decode_attention(synth.bf16_bits(q), bt.numpy(),
                                      np.array(seq, np.int32), pool,
                                      R_k.numpy(), R_v.numpy(), h_kv, win=win,
                                      win_slot=slots, sink=sink, recent=recent,
                                      mu=mu)
    kf, vf, qf = k.double().numpy(), v.double().numpy(), q.double().numpy()
    for b in range(len(seq)):
        for j in range(h_q):
            h = j // (h_q // h_kv)
            ref = oracle_mod.attention_dense(
                qf[b, j], kf[cu[b]:cu[b + 1], h], vf[cu[b]:cu[b + 1], h],
                R_k.numpy()[h], R_v.numpy()[h], mu[h].astype(np.float64),
                clip_k=0.96, clip_v=0.92, sink=sink, recent=recent, group=128)
            np.testing.assert_allclose(out[b, j], ref, atol=1e-12)


def test_unsupported_group_is_rejected(oracle_mod):
    with pytest.raises(ValueError):
        oracle_mod.rotate_quantize(np.zeros(D), EYE, group=64)
