"""Test infrastructure: OptR's offline rotation calibration, written out in
plain float64 PyTorch on the CPU.

This is the paper's one-time calibration (Sec. 4.2 "Orthogonal Rotation
Refinement", Sec. 4.3-4.4 the output-aware key and value objectives,
Sec. 4.5 "INT2-Aware Orthogonal Calibration" with its straight-through
estimator; Appendix, "OptR Algorithm"), run on synthetic traces: it
produces the {R_K, R_V, mu} per KV head that the cache write and the decode
take as inputs.  Only tests may import it; the library does not calibrate.

Every step follows the paper's notation:
  R_K = R_K^0 exp(A_K - A_K^T), R_V = R_V^0 exp(A_V - A_V^T)   (skew generators)
  effective keys   k~_s = Q2((k_s - mu) R_K) R_K^T   (window positions: k_s - mu)
  effective values v~_s = Q2(v_s R_V) R_V^T          (window positions: v_s)
  p_t      = softmax_{s<=t}(<q_t, k_s>/sqrt(d))       (BF16 reference)
  p_t^K    = softmax_{s<=t}(<q_t, k~_s>/sqrt(d))
  e_K(t,j) = [(p_t^K - p_t)^T V] W_{O,j}^T
  L_K      = mean_{t,j} KL(p_t || p_t^K) + lambda_K ||e_K||^2 / d_model
  e_V(t,j) = [phat_t^K^T (V~ - V)] W_{O,j}^T,  phat^K from the selected R_K
  L_V      = mean_{t,j} ||e_V||^2 / d_model
  Q2's gradient is the straight-through indicator of the clipping range.
Gradients are taken by torch.autograd (a library routine, through
torch.linalg.matrix_exp); Adam is written out.  Readings of the paper:
  * Q2 is the cache's quantizer (group-wise asymmetric INT2, codes from the
    clipped range, fp16-rounded scale and min), evaluated in float64;
  * the STE indicator 1{|Z| <= tau_c} is read as "inside the clipped range
    [c min, c max] of the value's group"; the group's range itself carries
    no gradient;
  * the window positions of query t are s < sink and s > t - recent;
  * the base rotation R^0 is the normalized Sylvester-Hadamard matrix.
"""
from __future__ import annotations

import math

import torch

F64 = torch.float64


def hadamard(d: int) -> torch.Tensor:
    """Normalized Sylvester-Hadamard matrix H / sqrt(d) (d a power of 2):
    an orthogonal base rotation R^0 (QuaRot's choice, Sec. 2)."""
    assert d > 0 and d & (d - 1) == 0
    H = torch.ones(1, 1, dtype=F64)
    while H.shape[0] < d:
        H = torch.cat([torch.cat([H, H], 1), torch.cat([H, -H], 1)], 0)
    return H / math.sqrt(d)


def rotation(R0: torch.Tensor, A: torch.Tensor) -> torch.Tensor:
    """R = R^0 exp(A - A^T): orthogonal for any A (Sec. 4.2)."""
    return R0 @ torch.linalg.matrix_exp(A - A.transpose(-1, -2))


def _f16(x: torch.Tensor) -> torch.Tensor:
    """The stored fp16 value of a float64 scale or min: rounded to float32,
    then to fp16 (both round-to-nearest-even), as the cache's quantizer
    stores the fp16 value of its float32 range.  Spelled out because a
    direct float64 -> fp16 conversion rounds once and can differ by an
    fp16 ulp."""
    return x.to(torch.float32).to(torch.float16).to(F64)


class Q2STE(torch.autograd.Function):
    """Group-wise INT2 quantize-dequantize of the rows of z (last dimension,
    groups of `group` channels), clipping ratio `clip`; backward passes the
    gradient where the value lies inside its group's clipped range."""

    @staticmethod
    def forward(ctx, z, clip, group):
        n, d = z.shape
        zg = z.reshape(n, d // group, group)
        mn = clip * zg.amin(dim=2, keepdim=True)
        mx = clip * zg.amax(dim=2, keepdim=True)
        r = mx - mn
        deg = ~(r > 1e-30)
        inv = torch.where(deg, torch.zeros_like(r), 3.0 / torch.where(deg, torch.ones_like(r), r))
        u = (torch.minimum(torch.maximum(zg, mn), mx) - mn) * inv
        codes = torch.clamp(torch.round(u), 0, 3)  # round half to even
        scale = torch.where(deg, torch.zeros_like(r), _f16(r / 3.0))
        zhat = codes * scale + _f16(mn)
        ctx.save_for_backward(((zg >= mn) & (zg <= mx)).reshape(n, d))
        return zhat.reshape(n, d)

    @staticmethod
    def backward(ctx, g):
        (inside,) = ctx.saved_tensors
        return g * inside.to(g.dtype), None, None


def q2(z, clip=1.0, group=32):
    return Q2STE.apply(z, clip, group)


def window_mask(T: int, t_pos: torch.Tensor, sink: int, recent: int) -> torch.Tensor:
    """[len(t_pos)][T] True where position s is a BF16 window position for
    the query at position t (s < sink or s > t - recent)."""
    s = torch.arange(T)
    return (s[None, :] < sink) | (s[None, :] > t_pos[:, None] - recent)


def _attention_probs(qh, keys, t_pos, scale):
    """softmax over s <= t of <q_t, keys_s> * scale; qh [nt][d], keys
    [nt][T][d] or [T][d]."""
    if keys.dim() == 2:
        logits = qh @ keys.T
    else:
        logits = torch.einsum("td,tsd->ts", qh, keys)
    T = logits.shape[1]
    causal = torch.arange(T)[None, :] <= t_pos[:, None]
    logits = torch.where(causal, logits * scale, torch.full_like(logits, -math.inf))
    return torch.softmax(logits, dim=1)


def effective_keys(K, mu, R_K, clip, group, win):
    """[nt][T][d]: quantized centered keys mapped back, exact centered keys
    at window positions (Sec. 4.1)."""
    kc = K - mu
    kq = q2(kc @ R_K, clip, group) @ R_K.T
    if win is None:
        return kq
    return torch.where(win[:, :, None], kc[None], kq[None])


def effective_values(V, R_V, clip, group, win):
    vq = q2(V @ R_V, clip, group) @ R_V.T
    if win is None:
        return vq
    return torch.where(win[:, :, None], V[None], vq[None])


def key_loss(q, K, V, mu, R_K, W_O, t_pos, lam=1.0, clip=1.0, group=32,
             sink=0, recent=0, quantize=True):
    """L_K (Sec. 4.3) for one KV head.  q [nt][g][d] (the g query heads of
    the group at positions t_pos), K, V [T][d], W_O [g][d_model][d]."""
    d = K.shape[1]
    scale = 1.0 / math.sqrt(d)
    win = window_mask(K.shape[0], t_pos, sink, recent) if sink or recent else None
    if quantize:
        kt = effective_keys(K, mu, R_K, clip, group, win)
    else:
        kt = (K - mu) @ R_K @ R_K.T
    total = 0.0
    n = 0
    for j in range(q.shape[1]):
        p = _attention_probs(q[:, j], K, t_pos, scale)
        pk = _attention_probs(q[:, j], kt, t_pos, scale)
        kl = (p * (torch.log(p.clamp_min(1e-300)) - torch.log(pk.clamp_min(1e-300)))).sum(1)
        e = ((pk - p) @ V) @ W_O[j].T
        total = total + (kl + lam * (e * e).sum(1) / W_O.shape[1]).sum()
        n += q.shape[0]
    return total / n


def value_loss(q, K, V, mu, R_K, R_V, W_O, t_pos, clip_k=1.0, clip_v=1.0,
               group=32, sink=0, recent=0, quantize=True):
    """L_V (Sec. 4.4) for one KV head, under the attention of the selected
    key rotation R_K (held fixed, no gradient)."""
    d = K.shape[1]
    scale = 1.0 / math.sqrt(d)
    win = window_mask(K.shape[0], t_pos, sink, recent) if sink or recent else None
    with torch.no_grad():
        kt = (effective_keys(K, mu, R_K, clip_k, group, win) if quantize
              else (K - mu) @ R_K @ R_K.T)
    if quantize:
        vt = effective_values(V, R_V, clip_v, group, win)
    else:
        vt = V @ R_V @ R_V.T
    total = 0.0
    n = 0
    for j in range(q.shape[1]):
        with torch.no_grad():
            ph = _attention_probs(q[:, j], kt, t_pos, scale)
        if vt.dim() == 2:
            diff = ph @ (vt - V)
        else:
            diff = torch.einsum("ts,tsd->td", ph, vt - V[None])
        e = diff @ W_O[j].T
        total = total + ((e * e).sum(1) / W_O.shape[1]).sum()
        n += q.shape[0]
    return total / n


class Adam:
    """Adam (Kingma & Ba) written out: m = b1 m + (1-b1) g,
    v = b2 v + (1-b2) g^2, x -= lr * mhat / (sqrt(vhat) + eps)."""

    def __init__(self, lr=0.02, b1=0.9, b2=0.999, eps=1e-8):
        self.lr, self.b1, self.b2, self.eps = lr, b1, b2, eps
        self.m = self.v = None
        self.t = 0

    def step(self, x: torch.Tensor, g: torch.Tensor) -> torch.Tensor:
        if self.m is None:
            self.m = torch.zeros_like(x)
            self.v = torch.zeros_like(x)
        self.t += 1
        self.m = self.b1 * self.m + (1 - self.b1) * g
        self.v = self.b2 * self.v + (1 - self.b2) * g * g
        mh = self.m / (1 - self.b1 ** self.t)
        vh = self.v / (1 - self.b2 ** self.t)
        return x - self.lr * mh / (vh.sqrt() + self.eps)


def calibrate_head(q, K, V, W_O, t_pos, R0_K=None, R0_V=None, steps=80,
                   lr=0.02, lam=1.0, clip_k=1.0, clip_v=1.0, group=32,
                   sink=0, recent=0, select_every=20, held_out=None):
    """The appendix algorithm for one KV head: mu from the trace's keys,
    A_K by Adam on L_K (values in BF16), then A_V by Adam on L_V under the
    selected key rotation.  Every `select_every` steps (and at step 0) the
    rotation is scored on the held-out trace (q, K, V, t_pos; the
    calibration trace when None) and the best one is kept (the paper's
    held-out selection every 20 steps).  Returns R_K, R_V, mu and the
    training-loss histories (the loss before each step)."""
    d = K.shape[1]
    R0_K = hadamard(d) if R0_K is None else R0_K
    R0_V = hadamard(d) if R0_V is None else R0_V
    mu = K.mean(0)
    hq, hK, hV, ht = held_out if held_out is not None else (q, K, V, t_pos)

    def run(loss_fn, R0):
        hist = []
        A = torch.zeros(d, d, dtype=F64)
        opt = Adam(lr)
        best_score, best_R = None, None
        for i in range(steps + 1):
            if i % select_every == 0 or i == steps:
                with torch.no_grad():
                    R = rotation(R0, A)
                    score = float(loss_fn(R, held=True))
                if best_score is None or score < best_score:
                    best_score, best_R = score, R
            if i == steps:
                break
            A.requires_grad_(True)
            loss = loss_fn(rotation(R0, A), held=False)
            (g,) = torch.autograd.grad(loss, A)
            hist.append(float(loss.detach()))
            A = opt.step(A.detach(), g)
        return best_R, hist

    def lk(R, held):
        a = (hq, hK, hV, ht) if held else (q, K, V, t_pos)
        return key_loss(a[0], a[1], a[2], mu, R, W_O, a[3], lam, clip_k, group,
                        sink, recent)

    R_K, hist_k = run(lk, R0_K)

    def lv(R, held):
        a = (hq, hK, hV, ht) if held else (q, K, V, t_pos)
        return value_loss(a[0], a[1], a[2], mu, R_K, R, W_O, a[3], clip_k,
                          clip_v, group, sink, recent)

    R_V, hist_v = run(lv, R0_V)
    return R_K, R_V, mu, hist_k, hist_v
