"""Pins of the CPU oracle to facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: hand-worked
values (tests/golden/), closed forms, exact invariances the paper states,
special cases that reduce to a library routine, or brute-force equivalences
between two differently written statements of the same formula.
"""
import os

import numpy as np
import pytest
import torch

from paper_2608_02691_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
D = 128


def _f16(bits):
    return float(np.array([bits], np.uint16).view(np.float16)[0])


def _bits(t):
    return synth.bf16_bits(t)


def _read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append([c.strip() for c in line.split("|")])
    return rows


# ------------------------------------------------------------- quantizer

def test_quantizer_hand_worked_groups(oracle_mod):
    """Sec. 3.1 (Q2, four levels, affine per group): hand-worked groups."""
    rows = _read_golden("quant_groups.txt")
    assert len(rows) >= 8
    for z, codes, scale, mn, byte, deg in rows:
        z = np.array([float(x) for x in z.split()], np.float32)
        want = [int(c) for c in codes.split()]
        c, s, m, u, d = oracle_mod.quantize_group(z)
        assert list(c) == want, (z, c)
        assert _f16(s) == float(scale)
        assert _f16(m) == float(mn)
        assert d == bool(int(deg))
        packed = sum(int(ci) << (2 * r) for r, ci in enumerate(c))
        assert packed == int(byte, 16)


def test_quantizer_32_group_is_tiled_rule(oracle_mod):
    """The 32-channel group follows the same rule as the 4-value cases."""
    for z, codes, scale, mn, _, _ in _read_golden("quant_groups.txt"):
        z4 = np.array([float(x) for x in z.split()], np.float32)
        c, s, m, _, _ = oracle_mod.quantize_group(np.tile(z4, 8))
        assert list(c) == [int(x) for x in codes.split()] * 8
        assert _f16(s) == float(scale) and _f16(m) == float(mn)


def test_quantizer_error_bound_and_monotone(oracle_mod):
    """Affine INT2 with rounding to nearest: |zhat - z| <= scale/2 up to the
    fp16 rounding of scale and min; codes are monotone in z and the group
    extremes map to levels 0 and 3."""
    rng = np.random.default_rng(1)
    for trial in range(400):
        z = (rng.standard_t(4, 32) * rng.uniform(0.01, 50)).astype(np.float32)
        c, s, m, u, deg = oracle_mod.quantize_group(z)
        assert not deg
        r = float(z.max()) - float(z.min())
        sc, mn = _f16(s), _f16(m)
        zhat = c.astype(np.float64) * sc + mn
        slack = 3 * abs(sc - r / 3) + abs(mn - float(z.min())) + 1e-6 * r
        assert np.all(np.abs(zhat - z) <= r / 6 + slack)
        order = np.argsort(z, kind="stable")
        assert np.all(np.diff(c[order].astype(int)) >= 0)
        assert c[np.argmin(z)] == 0 and c[np.argmax(z)] == 3


def test_quantizer_clip_saturates(oracle_mod):
    """Clipping ratio c < 1 narrows the range to [c*min, c*max]; values
    outside saturate at levels 0 and 3 (Sec. 3.1, Eq. 18's threshold tau_c
    bounds the representable range)."""
    z = np.array([-10, -1, 0, 1, 2, 10] + [0.5] * 26, np.float32)
    c, s, m, u, _ = oracle_mod.quantize_group(z, clip=0.5)
    assert _f16(m) == -5.0 and abs(_f16(s) - 10 / 3) < 2e-3
    assert c[0] == 0 and c[5] == 3
    c1, _, _, _, _ = oracle_mod.quantize_group(z, clip=1.0)
    assert c1[1] == 1 and c[1] == 1  # -1 -> u = 1.2 with clip 0.5


def test_quantizer_degenerate_group(oracle_mod):
    c, s, m, u, d = oracle_mod.quantize_group(np.full(32, -2.25, np.float32))
    assert d and not c.any() and s == 0 and _f16(m) == -2.25


# ------------------------------------------------------------ layout

def _identity(h_kv=1):
    return np.tile(np.eye(D, dtype=np.float32), (h_kv, 1, 1))


def test_slot_layout_golden(oracle_mod):
    """Byte order of a slot's codes and metadata, per the pool layout."""
    for name, formula, hexbytes in _read_golden("slot_layout.txt"):
        ch = np.arange(D)
        g, w, r = ch // 32, (ch % 32) // 4, ch % 4
        z = {"r": r, "(r+g)%4": (r + g) % 4, "(r+w)%4": (r + w) % 4}[formula]
        k = torch.tensor(z, dtype=torch.bfloat16).view(1, 1, D)
        pool = np.zeros((1, 1, 1536), np.uint8)
        oracle_mod.kv_append(_bits(k), _bits(k), [0, 1], [3], [[0]], pool,
                             _identity(), _identity(), np.zeros((1, D)))
        want = bytes.fromhex(hexbytes.replace(" ", ""))
        assert bytes(pool[0, 0, 3 * 32:4 * 32]) == want, name      # K slot 3
        assert bytes(pool[0, 0, 512 + 96:512 + 128]) == want, name  # V slot 3
        meta = bytes(pool[0, 0, 1024 + 48:1024 + 64])
        assert meta == bytes.fromhex("003c0000") * 4
        others = np.delete(pool[0, 0, :512].reshape(16, 32), 3, axis=0)
        assert not others.any()  # only slot 3 written


def test_compact_g128_record_golden(oracle_mod):
    """The compact G = 128 record (Sec. 5's one scale and min per 128
    channels): 1152 bytes per (page, KV head), codes laid out as with G = 32,
    one 4-byte (scale, min) per slot at 1024 (keys) and 1088 (values), and
    nothing else written."""
    meta = {name: (int(off), bytes.fromhex(hx.replace(" ", "")))
            for name, off, hx in _read_golden("slot_layout_g128.txt")}
    for name, formula, hexbytes in _read_golden("slot_layout.txt"):
        ch = np.arange(D)
        g, w, r = ch // 32, (ch % 32) // 4, ch % 4
        z = {"r": r, "(r+g)%4": (r + g) % 4, "(r+w)%4": (r + w) % 4}[formula]
        k = torch.tensor(z, dtype=torch.bfloat16).view(1, 1, D)
        pool = np.zeros((1, 1, 1152), np.uint8)
        oracle_mod.kv_append(_bits(k), _bits(k), [0, 1], [3], [[0]], pool,
                             _identity(), _identity(), np.zeros((1, D)),
                             group=128)
        want = bytes.fromhex(hexbytes.replace(" ", ""))
        assert bytes(pool[0, 0, 3 * 32:4 * 32]) == want, name
        assert bytes(pool[0, 0, 512 + 96:512 + 128]) == want, name
        for field, (off, val) in meta.items():
            assert bytes(pool[0, 0, off:off + len(val)]) == val, (name, field)
        rest = pool[0, 0].copy()
        rest[3 * 32:4 * 32] = 0
        rest[512 + 96:512 + 128] = 0
        for off, val in meta.values():
            rest[off:off + len(val)] = 0
        assert not rest.any(), name  # only slot 3's codes and pairs written
        kh, vh = oracle_mod.read_slot(pool, 0, 0, 3)
        assert np.array_equal(kh, z.astype(np.float64)), name
        assert np.array_equal(vh, z.astype(np.float64)), name


def test_rotation_is_right_multiplication(oracle_mod):
    """Row-vector convention z' = z R (Intro and Sec. 3.1 Eq. 4): with R a
    permutation matrix R[i][pi(i)] = 1, channel i lands on channel pi(i)."""
    rng = np.random.default_rng(2)
    pi = rng.permutation(D)
    R = np.zeros((D, D), np.float32)
    R[np.arange(D), pi] = 1.0
    x = rng.standard_normal(D)
    z, *_ = oracle_mod.rotate_quantize(x, R)
    assert np.array_equal(z[pi], x)


# ------------------------------------------------- attention special cases

def _sdpa(q, K, V):
    """torch's scaled_dot_product_attention in fp64 (library routine)."""
    out = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q).view(1, 1, 1, D), torch.tensor(K).view(1, 1, -1, D),
        torch.tensor(V).view(1, 1, -1, D))
    return out.view(D).numpy()


def _rand_case(rng, n):
    q = rng.standard_normal(D)
    K = rng.standard_t(4, (n, D)) + np.where(rng.random(D) < 0.03, 8.0, 0.0)
    V = rng.standard_t(4, (n, D))
    return q, K, V


def test_full_precision_identity_reduces_to_sdpa(oracle_mod):
    """Q2 = identity, R = I, mu = 0: Eq. 1-2 are plain scaled dot-product
    attention."""
    rng = np.random.default_rng(3)
    for n in (1, 2, 17, 300):
        q, K, V = _rand_case(rng, n)
        o = oracle_mod.attention_dense(q, K, V, np.eye(D), np.eye(D),
                                       np.zeros(D), quantize=False)
        np.testing.assert_allclose(o, _sdpa(q, K, V), rtol=0, atol=1e-12)


def test_full_precision_rotation_invariance(oracle_mod):
    """Sec. 3.1: with Q2 the identity, D_{R,c}(z) = z, so any orthogonal
    R_K, R_V leave the output unchanged."""
    rng = np.random.default_rng(4)
    Rk, Rv = synth.rotations_fp64(1, 5)
    Rk, Rv = Rk[0].numpy(), Rv[0].numpy()
    q, K, V = _rand_case(rng, 64)
    ref = _sdpa(q, K, V)
    o = oracle_mod.attention_dense(q, K, V, Rk.astype(np.float32),
                                   Rv.astype(np.float32), np.zeros(D),
                                   quantize=False)
    # the float32 cast of R is orthogonal to ~1e-7, which bounds the error
    np.testing.assert_allclose(o, ref, atol=5e-6 * np.abs(ref).max())


def test_full_precision_centering_invariance(oracle_mod):
    """Sec. 4.1: subtracting the same mu from every key shifts all logits of a
    query by one constant; softmax, hence the output, is unchanged."""
    rng = np.random.default_rng(6)
    q, K, V = _rand_case(rng, 50)
    mu = rng.standard_normal(D) * 5
    o0 = oracle_mod.attention_dense(q, K, V, np.eye(D), np.eye(D),
                                    np.zeros(D), quantize=False)
    o1 = oracle_mod.attention_dense(q, K, V, np.eye(D), np.eye(D), mu,
                                    quantize=False)
    np.testing.assert_allclose(o1, o0, atol=1e-12)


def test_single_token_closed_form(oracle_mod):
    """One cached token: softmax weight 1, so out = D_{R_V}(v) = vhat R_V^T."""
    rng = np.random.default_rng(7)
    q, K, V = _rand_case(rng, 1)
    o = oracle_mod.attention_dense(q, K, V, np.eye(D), np.eye(D), np.zeros(D))
    z, c, s, m, _ = oracle_mod.rotate_quantize(V[0], np.eye(D, dtype=np.float32))
    vhat = np.array([c[i] * _f16(s[i // 32]) + _f16(m[i // 32]) for i in range(D)])
    np.testing.assert_array_equal(o, vhat)


def test_two_equal_keys_average_values(oracle_mod):
    """Two identical keys get equal weight: out = (vbar_1 + vbar_2) / 2."""
    rng = np.random.default_rng(8)
    q, K, V = _rand_case(rng, 2)
    K[1] = K[0]
    o = oracle_mod.attention_dense(q, K, V, np.eye(D), np.eye(D), np.zeros(D))
    v0 = oracle_mod.attention_dense(q, K[:1], V[:1], np.eye(D), np.eye(D), np.zeros(D))
    v1 = oracle_mod.attention_dense(q, K[1:], V[1:], np.eye(D), np.eye(D), np.zeros(D))
    np.testing.assert_allclose(o, (v0 + v1) / 2, atol=1e-14)


def test_softmax_weights_sum_to_one_and_favour_aligned_key(oracle_mod):
    rng = np.random.default_rng(9)
    q, K, V = _rand_case(rng, 200)
    K[123] = q / np.linalg.norm(q) * 40.0
    _, p = oracle_mod.attention_dense(q, K, V, np.eye(D), np.eye(D),
                                      np.zeros(D), want_p=True)
    assert abs(p.sum() - 1) < 1e-12 and int(np.argmax(p)) == 123


# ------------------------------------------------- paged path equivalences

def _paged_case(rng, seq_tokens, h_kv=2, h_q=4, shuffle=True, seed=0):
    B = len(seq_tokens)
    R_k, R_v = synth.rotations(h_kv, seed)
    n = sum(seq_tokens)
    k = torch.tensor(rng.standard_t(4, (n, h_kv, D)) +
                     np.where(rng.random((1, h_kv, D)) < 0.03, 8.0, 0.0),
                     dtype=torch.bfloat16)
    v = torch.tensor(rng.standard_t(4, (n, h_kv, D)), dtype=torch.bfloat16)
    q = torch.tensor(rng.standard_normal((B, h_q, D)), dtype=torch.bfloat16)
    mu = synth.key_mean(k)
    bt, num_pages = synth.page_tables(seq_tokens, shuffle, seed)
    cu = np.concatenate([[0], np.cumsum(seq_tokens)]).astype(np.int32)
    pool = np.zeros((num_pages, h_kv, 1536), np.uint8)
    return dict(k=k, v=v, q=q, mu=mu.numpy(), R_k=R_k.numpy(),
                R_v=R_v.numpy(), bt=bt.numpy(), cu=cu, pool=pool,
                seq=np.array(seq_tokens, np.int32), h_kv=h_kv, h_q=h_q)


def _fill(oracle_mod, c):
    oracle_mod.kv_append(_bits(c["k"]), _bits(c["v"]), c["cu"],
                         np.zeros(len(c["seq"]), np.int32), c["bt"], c["pool"],
                         c["R_k"], c["R_v"], c["mu"])


def test_rotated_query_form_equals_inverse_rotation_form(oracle_mod):
    """Appendix, "Rotated-query implementation" and "Equivalent Inference
    Implementation": q (k_R R_K^T)^T = (q R_K) k_R^T and o = o' R_V^T, so the
    paged decode (rotated query, rotated output) equals the dense statement
    that maps every dequantized key and value back with R^T (Eq. 4)."""
    rng = np.random.default_rng(10)
    seq = [1, 2, 15, 16, 17, 33]
    c = _paged_case(rng, seq, shuffle=True)
    _fill(oracle_mod, c)
    out = oracle_mod.decode_attention(_bits(c["q"]), c["bt"], c["seq"],
                                      c["pool"], c["R_k"], c["R_v"], c["h_kv"])
    ratio = c["h_q"] // c["h_kv"]
    kf = c["k"].to(torch.float64).numpy()
    vf = c["v"].to(torch.float64).numpy()
    qf = c["q"].to(torch.float64).numpy()
    for b in range(len(seq)):
        s0, s1 = c["cu"][b], c["cu"][b + 1]
        for j in range(c["h_q"]):
            h = j // ratio
            ref = oracle_mod.attention_dense(
                qf[b, j], kf[s0:s1, h], vf[s0:s1, h], c["R_k"][h],
                c["R_v"][h], c["mu"][h].astype(np.float64))
            np.testing.assert_allclose(out[b, j], ref, atol=1e-12)


def test_physical_page_order_is_irrelevant(oracle_mod):
    """The block table only relocates pages: shuffled and in-order pools give
    bit-identical outputs."""
    rng = np.random.default_rng(11)
    seq = [40, 5, 64]
    outs = []
    for shuffle in (False, True):
        r = np.random.default_rng(11)
        c = _paged_case(r, seq, shuffle=shuffle)
        _fill(oracle_mod, c)
        outs.append(oracle_mod.decode_attention(
            _bits(c["q"]), c["bt"], c["seq"], c["pool"], c["R_k"], c["R_v"],
            c["h_kv"]))
    np.testing.assert_array_equal(outs[0], outs[1])


def test_centering_is_applied_before_quantization(oracle_mod):
    """Sec. 4.1: the stored key is Q2((k - mu) R_K).  Appending k with mean mu
    must store exactly what appending (k - mu) with mean 0 stores (inputs
    chosen so that k - mu is exact in bf16)."""
    rng = np.random.default_rng(12)
    m = rng.integers(-64, 65, (8, 1, D))
    k = torch.tensor(m / 16.0, dtype=torch.bfloat16)
    mu = np.where(rng.random((1, D)) < 0.1, 8.0, 0.0).astype(np.float32)
    kc = torch.tensor(m / 16.0 - mu[None], dtype=torch.bfloat16)
    assert torch.equal(kc.double(), k.double() - torch.tensor(mu[None], dtype=torch.float64))
    R_k, R_v = synth.rotations(1, 3)
    bt = np.zeros((1, 1), np.int32)
    p1 = np.zeros((1, 1, 1536), np.uint8)
    p2 = np.zeros((1, 1, 1536), np.uint8)
    oracle_mod.kv_append(_bits(k), _bits(k), [0, 8], [0], bt, p1, R_k, R_v, mu)
    oracle_mod.kv_append(_bits(kc), _bits(k), [0, 8], [0], bt, p2, R_k, R_v,
                         np.zeros((1, D), np.float32))
    np.testing.assert_array_equal(p1, p2)
    # and centering matters: without mu the stored keys differ
    p3 = np.zeros((1, 1, 1536), np.uint8)
    oracle_mod.kv_append(_bits(k), _bits(k), [0, 8], [0], bt, p3, R_k, R_v,
                         np.zeros((1, D), np.float32))
    assert not np.array_equal(p1[..., :512], p3[..., :512])


def test_centering_reduces_key_reconstruction_error(oracle_mod):
    """Sec. 4.1: large channel-wise key offsets widen the INT2 range;
    subtracting the per-channel mean before rotation shrinks the rotated
    reconstruction error (norms are preserved by R, so the rotated-space
    error is the key error)."""
    rng = np.random.default_rng(13)
    Rk, _ = synth.rotations(1, 1)
    R = Rk[0].numpy()
    off = np.zeros(D)
    off[rng.choice(D, 4, replace=False)] = rng.choice([-1, 1], 4) * rng.uniform(6, 10, 4)
    K = rng.standard_t(4, (200, D)) + off
    mu = K.mean(0)

    def err(x):
        z, c, s, m, _ = oracle_mod.rotate_quantize(x, R)
        zhat = np.array([c[i] * _f16(s[i // 32]) + _f16(m[i // 32]) for i in range(D)])
        return np.linalg.norm(zhat - z)

    e_plain = np.mean([err(k) for k in K])
    e_cent = np.mean([err(k - mu) for k in K])
    assert e_cent < 0.8 * e_plain


def test_zero_length_and_out_of_range(oracle_mod):
    rng = np.random.default_rng(14)
    c = _paged_case(rng, [16, 3])
    _fill(oracle_mod, c)
    seq = np.array([0, 3], np.int32)
    out = oracle_mod.decode_attention(_bits(c["q"]), c["bt"], seq, c["pool"],
                                      c["R_k"], c["R_v"], c["h_kv"])
    assert not out[0].any() and out[1].any()
    bad = c["bt"].copy()
    bad[1, 0] = 10_000
    with pytest.raises(ValueError):
        oracle_mod.decode_attention(_bits(c["q"]), bad, seq, c["pool"],
                                    c["R_k"], c["R_v"], c["h_kv"])


# ------------------------------------------------- synthetic inputs

def test_generated_rotations_are_orthogonal():
    Rk, Rv = synth.rotations_fp64(8, 0)
    eye = torch.eye(D, dtype=torch.float64)
    for R in (Rk, Rv):
        assert (R @ R.transpose(1, 2) - eye).abs().max() < 1e-12
        assert torch.all(torch.diagonal(torch.linalg.qr(R[0])[1]).abs() > 0)
    Rk32, _ = synth.rotations(8, 0)
    assert (Rk32.double() @ Rk32.double().transpose(1, 2) - eye).abs().max() < 1e-6


def test_needle_has_requested_cosine():
    wl = synth.workload("long128k", scale=1 / 64)
    case = synth.build_case(wl, seed=0)
    ratio = case["h_q"] // case["h_kv"]
    for h, pos in enumerate(case["needle"].tolist()):
        kc = case["k_ctx"][pos, h].double() - case["mu"][h].double()
        qv = case["q"][0, h * ratio].double()
        cos = float(kc @ qv / kc.norm() / qv.norm())
        assert abs(cos - 0.9) < 0.01


def test_group_boundaries_in_128_vector(oracle_mod):
    """Groups are 32 consecutive rotated channels, each with its own scale and
    min (Sec. 3.1, group size G).  Group g holds (g+1)*{0,1} in its first 16
    channels and (g+1)*{2,3} in its last 16, offset by 10g: with G = 32 the
    codes are 0/1 then 2/3, scale g+1, min 10g (a 16-wide grouping would give
    codes 0/3 only)."""
    ch = np.arange(D)
    g, r, half = ch // 32, ch % 4, (ch % 32) // 16
    level = np.where(half == 0, r % 2, 2 + r % 2)
    z = (g + 1) * level + 10.0 * g
    _, c, s, m, _ = oracle_mod.rotate_quantize(z, np.eye(D, dtype=np.float32))
    assert np.array_equal(c, level)
    assert [_f16(x) for x in s] == [1.0, 2.0, 3.0, 4.0]
    assert [_f16(x) for x in m] == [0.0, 10.0, 20.0, 30.0]
