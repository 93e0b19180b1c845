"""Pins of the calibration oracle (oracle/calibration.py: Sec. 4.2-4.5 and
the appendix algorithm) against facts that do not come from it: a library
Hadamard matrix, orthogonality of exp of a skew matrix, the cache quantizer
of the C oracle, the STE's indicator, exact zero losses when Q2 is the
identity, Adam's first step in closed form, finite differences of the loss
under the STE's surrogate, and that a short calibration lowers both losses.
"""
import math

import numpy as np
import pytest
import torch

from oracle import calibration as cal

D = 128
F64 = torch.float64


def test_hadamard_is_the_library_matrix():
    scipy_linalg = pytest.importorskip("scipy.linalg")
    for d in (2, 16, 128):
        H = cal.hadamard(d)
        ref = torch.tensor(scipy_linalg.hadamard(d), dtype=F64) / math.sqrt(d)
        assert torch.equal(H, ref)
        assert torch.allclose(H @ H.T, torch.eye(d, dtype=F64), atol=1e-14)


def test_exp_of_skew_generator_is_orthogonal():
    """Sec. 4.2: S = A - A^T is skew-symmetric, exp(S) orthogonal; A = 0
    leaves the base rotation."""
    g = torch.Generator().manual_seed(1)
    R0 = cal.hadamard(D)
    for s in (0.0, 0.01, 0.3):
        A = torch.randn(D, D, generator=g, dtype=F64) * s
        R = cal.rotation(R0, A)
        assert torch.allclose(R @ R.T, torch.eye(D, dtype=F64), atol=1e-12)
    assert torch.equal(cal.rotation(R0, torch.zeros(D, D, dtype=F64)), R0)


@pytest.mark.parametrize("group,clip", [(32, 1.0), (128, 0.96), (128, 0.92)])
def test_q2_forward_is_the_cache_quantizer(oracle_mod, group, clip):
    """The calibration's Q2 dequantizes exactly as the cache's quantizer
    (the C oracle; decisions there in float32, here in float64: agreement
    outside ~1e-7 of a rounding boundary)."""
    g = np.random.default_rng(2)
    Z = g.standard_t(4, (200, D)) * g.uniform(0.2, 5.0, (200, 1))
    got = cal.q2(torch.tensor(Z), clip, group).numpy()
    eye = np.eye(D, dtype=np.float32)
    bad = 0
    for i in range(Z.shape[0]):
        z32 = Z[i].astype(np.float32).astype(np.float64)  # what the C side sees
        _, codes, s, m, _ = oracle_mod.rotate_quantize(z32, eye, clip, group=group)
        f16 = lambda b: float(np.array([b], np.uint16).view(np.float16)[0])
        ref = np.array([codes[c] * f16(s[c // 32]) + f16(m[c // 32]) for c in range(D)])
        bad += int((np.abs(got[i] - ref) > 1e-3 * np.abs(ref).max()).sum())
    assert bad <= 2, bad


def test_ste_passes_the_gradient_inside_the_clipped_range():
    """Sec. 4.5: dQ2/dZ ~ 1{inside the clipping range}, elementwise."""
    g = torch.Generator().manual_seed(3)
    Z = torch.randn(50, D, generator=g, dtype=F64).requires_grad_(True)
    up = torch.randn(50, D, generator=g, dtype=F64)
    clip = 0.9
    out = cal.q2(Z, clip, 32)
    (grad,) = torch.autograd.grad((out * up).sum(), Z)
    zg = Z.detach().reshape(50, 4, 32)
    lo = clip * zg.amin(2, keepdim=True)
    hi = clip * zg.amax(2, keepdim=True)
    inside = ((zg >= lo) & (zg <= hi)).reshape(50, D)
    assert torch.equal(grad, up * inside)
    assert inside.float().mean() < 1.0  # clipping actually excludes values


def _trace(seed, T=192, g=4, d_model=64, offsets=True):
    gen = torch.Generator().manual_seed(seed)
    K = torch.distributions.StudentT(4.0).sample((T, D)).to(F64)
    if offsets:
        ch = torch.randperm(D, generator=gen)[:4]
        K[:, ch] += 8.0
    V = torch.distributions.StudentT(4.0).sample((T, D)).to(F64)
    t_pos = torch.arange(T - 32, T)
    q = torch.randn(len(t_pos), g, D, generator=gen, dtype=F64)
    W_O = torch.randn(g, d_model, D, generator=gen, dtype=F64) / math.sqrt(g * D)
    return q, K, V, W_O, t_pos


def test_losses_vanish_when_q2_is_the_identity():
    """With Q2 the identity the effective keys are k - mu and the values v
    for any rotation (Sec. 3.1): p^K = p (a constant logit shift), so both
    losses are zero up to rounding."""
    torch.manual_seed(4)
    q, K, V, W_O, t_pos = _trace(4)
    mu = K.mean(0)
    R = cal.rotation(cal.hadamard(D), torch.randn(D, D, dtype=F64) * 0.1)
    lk = cal.key_loss(q, K, V, mu, R, W_O, t_pos, quantize=False)
    lv = cal.value_loss(q, K, V, mu, R, R, W_O, t_pos, quantize=False)
    assert abs(float(lk)) < 1e-12 and abs(float(lv)) < 1e-24
    assert float(cal.key_loss(q, K, V, mu, R, W_O, t_pos)) > 1e-6


def test_adam_first_step_closed_form():
    """Adam's bias-corrected first step is lr * g / (|g| + eps)."""
    g = torch.tensor([0.5, -2.0, 1e-3, 0.0], dtype=F64)
    x0 = torch.tensor([1.0, 1.0, 1.0, 1.0], dtype=F64)
    opt = cal.Adam(lr=0.02)
    x1 = opt.step(x0, g)
    assert torch.allclose(x1, x0 - 0.02 * g / (g.abs() + 1e-8), rtol=0, atol=1e-15)


def test_gradient_matches_finite_differences_of_the_ste_surrogate():
    """The STE gradient is the exact gradient of the surrogate
    zhat(z) = zhat(z0) + 1{inside}(z - z0) around the current point; central
    differences of L_K built on that surrogate along a random direction
    match <dL/dA, dA> (rotation exponential, both uses of R and the two loss
    terms all enter)."""
    torch.manual_seed(5)
    q, K, V, W_O, t_pos = _trace(5, T=96)
    mu = K.mean(0)
    R0 = cal.hadamard(D)
    A0 = torch.randn(D, D, dtype=F64) * 0.05
    z0 = ((K - mu) @ cal.rotation(R0, A0)).detach()
    zhat0 = cal.q2(z0, 1.0, 32).detach()
    zg = z0.reshape(-1, 4, 32)
    inside = ((zg >= zg.amin(2, keepdim=True)) & (zg <= zg.amax(2, keepdim=True))).reshape(z0.shape)
    orig = cal.q2
    cal.q2 = lambda z, clip, group: zhat0 + inside * (z - z0)
    try:
        A = A0.clone().requires_grad_(True)
        L = cal.key_loss(q, K, V, mu, cal.rotation(R0, A), W_O, t_pos)
        (grad,) = torch.autograd.grad(L, A)
        dA = torch.randn(D, D, dtype=F64)
        eps = 1e-6
        lp = cal.key_loss(q, K, V, mu, cal.rotation(R0, A0 + eps * dA), W_O, t_pos)
        lm = cal.key_loss(q, K, V, mu, cal.rotation(R0, A0 - eps * dA), W_O, t_pos)
        fd = (float(lp) - float(lm)) / (2 * eps)
        an = float((grad * dA).sum())
        assert abs(fd - an) <= 1e-6 * max(abs(an), 1e-12), (fd, an)
    finally:
        cal.q2 = orig


def test_short_calibration_lowers_both_losses():
    """The appendix algorithm on a synthetic trace with outlier key
    channels (G = 32, small steps to keep it quick and monotone): Adam from
    the Hadamard base lowers L_K and L_V, and the rotations stay
    orthogonal."""
    torch.manual_seed(6)
    q, K, V, W_O, t_pos = _trace(6)
    R_K, R_V, mu, hk, hv = cal.calibrate_head(q, K, V, W_O, t_pos, steps=12,
                                              lr=0.001, select_every=4)
    assert hk[-1] < 0.9 * hk[0] and hv[-1] < 0.9 * hv[0], (hk, hv)
    for R in (R_K, R_V):
        assert torch.allclose(R @ R.T, torch.eye(D, dtype=F64), atol=1e-10)
    assert torch.equal(mu, K.mean(0))


def test_selection_keeps_the_best_scored_rotation():
    """Held-out selection (every 20 steps in the paper) includes the start:
    the selected key rotation scores no worse on the held-out trace than
    the base rotation, even with the paper's lr = 0.02."""
    torch.manual_seed(7)
    q, K, V, W_O, t_pos = _trace(7)
    t8 = _trace(8)
    ho = (t8[0], t8[1], t8[2], t8[4])  # q, K, V, query positions
    R_K, _, mu, _, _ = cal.calibrate_head(q, K, V, W_O, t_pos, steps=8,
                                          lr=0.02, select_every=4,
                                          held_out=ho)
    base = cal.key_loss(ho[0], ho[1], ho[2], mu, cal.hadamard(D), W_O, ho[3])
    got = cal.key_loss(ho[0], ho[1], ho[2], mu, R_K, W_O, ho[3])
    assert float(got) <= float(base)


def test_all_window_positions_make_both_losses_zero():
    """Window positions skip INT2 (Sec. 4.1, appendix: sink and recent
    tokens keep exact centered keys and exact values): with the windows
    covering every position both losses are zero whatever the rotation."""
    torch.manual_seed(9)
    q, K, V, W_O, t_pos = _trace(9, T=96)
    mu = K.mean(0)
    R = cal.rotation(cal.hadamard(D), torch.randn(D, D, dtype=F64) * 0.1)
    lk = cal.key_loss(q, K, V, mu, R, W_O, t_pos, sink=32, recent=96)
    lv = cal.value_loss(q, K, V, mu, R, R, W_O, t_pos, sink=32, recent=96)
    assert abs(float(lk)) < 1e-12 and float(lv) == 0.0
    # a window that leaves INT2 positions: the losses come back
    assert float(cal.key_loss(q, K, V, mu, R, W_O, t_pos, sink=16, recent=8)) > 1e-6
