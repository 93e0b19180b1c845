"""Pins of the oracle's BF16 windows (Sec. 3.1 opening paragraph: INT2 long
history with a small BF16 window; Sec. 4.1: sink and recent tokens stay in
BF16 with the same key centering; Sec. 5 "Implementation Details": 64 sink
and 256 recent tokens) against facts that do not come from the oracle:

* every position a window position: plain scaled dot-product attention on
  the raw bf16 keys and values (torch, fp64), whatever the pool holds;
* Q2 the identity: plain attention again for any mix of window and INT2
  positions, any orthogonal rotation and any key mean;
* the paged decode, fed through the window store by a multi-call cache
  write, equals the dense statement that marks window positions directly;
* the store rows follow the layout of include/optr.h.
"""
import numpy as np
import pytest
import torch

from paper_2608_02691_gb300 import synth

D = 128


def _bits(t):
    return synth.bf16_bits(t)


def _sdpa(q, K, V):
    """torch's scaled_dot_product_attention in fp64 (library routine)."""
    out = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q).view(1, 1, 1, D), torch.tensor(K).view(1, 1, -1, D),
        torch.tensor(V).view(1, 1, -1, D))
    return out.view(D).numpy()


def _history(rng, seq_tokens, calls, h_kv=2, h_q=8, seed=0, sink=16,
             recent=32, shuffle=True):
    """Sequences of seq_tokens tokens written by len(calls) cache writes:
    call c appends calls[c][b] tokens to sequence b (the calls of a sequence
    sum to its length).  Returns the oracle's pool and window store and the
    raw tokens per sequence."""
    B = len(seq_tokens)
    calls = [np.asarray(c, np.int64) for c in calls]
    assert np.array_equal(np.sum(calls, axis=0), seq_tokens)
    R_k, R_v = synth.rotations(h_kv, seed)
    toks_k, toks_v = [], []
    for n in seq_tokens:
        toks_k.append(torch.tensor(rng.standard_t(4, (n, h_kv, D)) +
                                   np.where(rng.random((1, h_kv, D)) < 0.03,
                                            8.0, 0.0), dtype=torch.bfloat16))
        toks_v.append(torch.tensor(rng.standard_t(4, (n, h_kv, D)),
                                   dtype=torch.bfloat16))
    mu = synth.key_mean(torch.cat(toks_k)).numpy()
    q = torch.tensor(rng.standard_normal((B, h_q, D)), dtype=torch.bfloat16)
    bt, num_pages = synth.page_tables(list(seq_tokens), shuffle, seed)
    bt = bt.numpy()
    pool = np.zeros((num_pages, h_kv, 1536), np.uint8)
    n_slots = B + 3
    slots = rng.permutation(n_slots)[:B].astype(np.int32)
    win = np.zeros((n_slots, h_kv, 2, sink + recent, D), np.uint16)
    done = np.zeros(B, np.int64)
    from oracle import oracle
    for c in calls:
        ks = [toks_k[b][done[b]:done[b] + c[b]] for b in range(B)]
        vs = [toks_v[b][done[b]:done[b] + c[b]] for b in range(B)]
        k = torch.cat(ks)
        v = torch.cat(vs)
        cu = np.concatenate([[0], np.cumsum(c)]).astype(np.int32)
        pos0 = done.astype(np.int32)
        if k.shape[0]:
            oracle.kv_append(_bits(k), _bits(v), cu, pos0, bt, pool, R_k.numpy(),
                             R_v.numpy(), mu)
            oracle.window_write(_bits(k), _bits(v), cu, pos0, win, slots, sink,
                                recent)
        done += c
    return dict(q=q, k=toks_k, v=toks_v, mu=mu, R_k=R_k.numpy(),
                R_v=R_v.numpy(), bt=bt, pool=pool, win=win, slots=slots,
                seq=np.array(seq_tokens, np.int32), h_kv=h_kv, h_q=h_q,
                sink=sink, recent=recent)


def _decode(oracle_mod, c, pool=None):
    return oracle_mod.decode_attention(
        _bits(c["q"]), c["bt"], c["seq"], c["pool"] if pool is None else pool,
        c["R_k"], c["R_v"], c["h_kv"], win=c["win"], win_slot=c["slots"],
        sink=c["sink"], recent=c["recent"], mu=c["mu"])


def test_all_window_positions_is_plain_attention(oracle_mod):
    """n <= sink + recent: every position is BF16, so the output is plain
    attention on the raw keys and values (the key centering shifts every
    logit of a query by one constant), and the INT2 pool is never read."""
    rng = np.random.default_rng(31)
    seq = [1, 7, 16, 40, 48]  # sink 16 + recent 32 = 48
    c = _history(rng, seq, [[1, 3, 16, 20, 30], [0, 4, 0, 20, 18]])
    pool = np.random.default_rng(1).integers(0, 256, c["pool"].shape, np.uint8)
    out = _decode(oracle_mod, c, pool)
    ratio = c["h_q"] // c["h_kv"]
    for b, n in enumerate(seq):
        K = c["k"][b].double().numpy()
        V = c["v"][b].double().numpy()
        for j in range(c["h_q"]):
            ref = _sdpa(c["q"][b, j].double().numpy(), K[:, j // ratio],
                        V[:, j // ratio])
            np.testing.assert_allclose(out[b, j], ref, rtol=0, atol=1e-12)


def test_identity_q2_with_windows_is_plain_attention(oracle_mod):
    """Q2 the identity (Sec. 3.1: then D_{R,c}(z) = z): whichever positions
    are windows, the dense statement is plain attention on (k, v), for an
    orthogonal rotation and a large key mean."""
    rng = np.random.default_rng(32)
    Rk, Rv = synth.rotations_fp64(1, 7)
    Rk, Rv = Rk[0].numpy().astype(np.float32), Rv[0].numpy().astype(np.float32)
    q = rng.standard_normal(D)
    n = 200
    K = rng.standard_t(4, (n, D)) + np.where(rng.random(D) < 0.05, 9.0, 0.0)
    V = rng.standard_t(4, (n, D))
    mu = K.mean(axis=0) + rng.standard_normal(D)
    ref = _sdpa(q, K, V)
    for sink, recent in ((0, 0), (16, 0), (0, 64), (64, 32), (128, 128)):
        o = oracle_mod.attention_dense(q, K, V, Rk, Rv, mu, quantize=False,
                                       sink=sink, recent=recent)
        # the float32 cast of R is orthogonal to ~1e-7
        np.testing.assert_allclose(o, ref, atol=5e-6 * np.abs(ref).max())


def test_window_keys_are_centered_like_int2_keys(oracle_mod):
    """Sec. 4.1 centers the BF16 keys by the same mu.  With Q2 active and a
    key mean of size ~9 on a few channels, leaving the window keys
    uncentered (k instead of k - mu) moves their logits by -<q, mu>/sqrt(d)
    relative to the INT2 keys and changes the output by far more than
    rounding; the oracle's window result matches the centered statement
    computed here from its parts."""
    rng = np.random.default_rng(33)
    n, sink, recent = 120, 16, 32
    q = rng.standard_normal(D)
    K = rng.standard_t(4, (n, D)) + np.where(rng.random(D) < 0.05, 9.0, 0.0)
    V = rng.standard_t(4, (n, D))
    mu = K.mean(axis=0)
    eye = np.eye(D, dtype=np.float32)
    o = oracle_mod.attention_dense(q, K, V, eye, eye, mu, sink=sink,
                                   recent=recent)
    # the same from its parts: window positions exact, INT2 positions the
    # dequantized (k - mu) / v of the single-token quantizer
    kbar = K - mu
    vbar = V.copy()
    for s in range(sink, n - recent):
        _, ck, sk, mk, _ = oracle_mod.rotate_quantize(K[s] - mu, eye)
        _, cv, sv, mv, _ = oracle_mod.rotate_quantize(V[s], eye)
        f16 = lambda b: float(np.array([b], np.uint16).view(np.float16)[0])
        kbar[s] = [ck[i] * f16(sk[i // 32]) + f16(mk[i // 32]) for i in range(D)]
        vbar[s] = [cv[i] * f16(sv[i // 32]) + f16(mv[i // 32]) for i in range(D)]
    a = kbar @ q / np.sqrt(D)
    p = np.exp(a - a.max())
    p /= p.sum()
    np.testing.assert_allclose(o, p @ vbar, atol=1e-12)
    # uncentered window keys would give a visibly different result
    kun = kbar.copy()
    win = np.r_[0:sink, n - recent:n]
    kun[win] = K[win]
    a2 = kun @ q / np.sqrt(D)
    p2 = np.exp(a2 - a2.max())
    p2 /= p2.sum()
    assert np.abs(p2 @ vbar - o).max() > 1e-3 * np.abs(o).max()


@pytest.mark.parametrize("shuffle", [False, True])
def test_paged_windows_equal_dense_windows(oracle_mod, shuffle):
    """Appendix, rotated-query and equivalent inference implementations,
    with windows: the paged decode (window positions from the store written
    over several cache writes, INT2 positions from the pool) equals the
    dense statement that marks the window positions directly."""
    rng = np.random.default_rng(34)
    # lengths below, at and above sink (16), sink + recent (48), ragged
    seq = [5, 16, 30, 48, 49, 77, 160, 203]
    calls = [[5, 16, 10, 40, 20, 60, 100, 3],
             [0, 0, 1, 1, 1, 1, 1, 1],
             [0, 0, 19, 7, 28, 16, 59, 199]]
    c = _history(rng, seq, calls, shuffle=shuffle)
    out = _decode(oracle_mod, c)
    ratio = c["h_q"] // c["h_kv"]
    for b in range(len(seq)):
        K = c["k"][b].double().numpy()
        V = c["v"][b].double().numpy()
        for j in range(c["h_q"]):
            h = j // ratio
            ref = oracle_mod.attention_dense(
                c["q"][b, j].double().numpy(), K[:, h], V[:, h], c["R_k"][h],
                c["R_v"][h], c["mu"][h].astype(np.float64), sink=c["sink"],
                recent=c["recent"])
            np.testing.assert_allclose(out[b, j], ref, atol=1e-12)


def test_window_positions_ignore_the_pool(oracle_mod):
    """Window positions are never read from the INT2 pool: overwriting
    their slots with random bytes leaves the output bit-identical."""
    rng = np.random.default_rng(35)
    seq = [100, 61]
    c = _history(rng, seq, [[60, 61], [40, 0]], shuffle=True)
    ref = _decode(oracle_mod, c)
    pool = c["pool"].copy()
    g = np.random.default_rng(2)
    for b, n in enumerate(seq):
        for s in list(range(c["sink"])) + list(range(n - c["recent"], n)):
            page = c["bt"][b, s // 16]
            for h in range(c["h_kv"]):
                for base, width in ((0, 32), (512, 32), (1024, 16), (1280, 16)):
                    off = base + (s % 16) * width
                    pool[page, h, off:off + width] = g.integers(0, 256, width)
    np.testing.assert_array_equal(_decode(oracle_mod, c, pool), ref)


def test_store_rows_follow_the_layout(oracle_mod):
    """include/optr.h: position s < sink in row s, later positions in row
    sink + (s - sink) % recent; after the writes, every window position of
    the final length sits in its row, keys in plane 0 and values in 1."""
    rng = np.random.default_rng(36)
    seq = [150, 20, 47]
    c = _history(rng, seq, [[100, 10, 47], [1, 10, 0], [49, 0, 0]])
    sink, recent = c["sink"], c["recent"]
    for b, n in enumerate(seq):
        kb, vb = _bits(c["k"][b]), _bits(c["v"][b])
        st = c["win"][c["slots"][b]]
        for s in range(n):
            if not (s < sink or s >= n - recent):
                continue
            row = s if s < sink else sink + (s - sink) % recent
            np.testing.assert_array_equal(st[:, 0, row], kb[s])
            np.testing.assert_array_equal(st[:, 1, row], vb[s])


def test_window_edge_cases(oracle_mod):
    """Zero-length sequences give zeros; a window slot out of range is an
    error."""
    rng = np.random.default_rng(37)
    c = _history(rng, [0, 20], [[0, 20]])
    out = _decode(oracle_mod, c)
    assert not out[0].any() and out[1].any()
    c["slots"] = np.array([0, c["win"].shape[0]], np.int32)
    with pytest.raises(ValueError):
        _decode(oracle_mod, c)
