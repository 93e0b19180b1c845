"""Seeded synthetic inputs for the rotated INT2 paged KV-cache path.

This module only draws random numbers and builds page tables; it holds none
of the method's arithmetic (no rotation, quantization or attention).  Both
the CUDA library's tests/benchmark and the CPU oracle are fed from it.

The five workloads mirror the paper's serving setting (Qwen3-8B-shaped GQA
layer: 32 query heads, 8 KV heads, head dim 128) with synthetic stand-ins for
the paper's model traces, which are not available:

  tiny      B=1, context 1024, K/V ~ N(0,1), pages in order.
  decode8k  B=16, context 8192, K/V Student-t (nu=4), pages shuffled.
  long128k  B=1, context 131072, Student-t, shuffled, one planted needle key
            per KV head (cosine 0.9 with the group's first query head).
  prefill   append of 4 x 32768 tokens, Student-t, shuffled tables.
  ragged    B=128, context ~ U[1024, 32768] per sequence, Student-t, pages
            randomly interleaved across sequences, plus one appended token
            per sequence.

Keys get a constant offset ~ sign * U(6, 10) on 4 random channels per KV head
(the channel-wise key offsets that motivate centering, Sec. 4.1); mu is the
float64 per-channel mean of the generated keys, stored as float32.  R_k and
R_v per KV head come from the QR decomposition of a seeded Gaussian 128x128
matrix, with column signs fixed so that diag(R_qr) > 0.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import torch

D = 128
PAGE = 16
_CHUNK = 1 << 25  # elements drawn per random call (bounds temporary memory)


@dataclass
class Workload:
    name: str
    B: int
    ctx: list            # cached tokens per sequence before the step
    dist: str            # "normal" or "t4"
    shuffle: bool        # shuffle physical pages
    needle: bool = False
    append: int = 0      # new tokens per sequence appended by the step
    h_q: int = 32
    h_kv: int = 8
    extra: dict = field(default_factory=dict)

    @property
    def n_ctx_tokens(self) -> int:
        return int(sum(self.ctx))


def workload(name: str, seed: int = 0, scale: float = 1.0) -> Workload:
    """The named workload; ``scale`` < 1 shrinks context lengths (parity cases
    that the oracle finishes in seconds) while keeping every structure."""
    def sc(n):
        return max(1, int(round(n * scale)))

    if name == "tiny":
        return Workload(name, 1, [sc(1024)], "normal", shuffle=False)
    if name == "decode8k":
        return Workload(name, 16, [sc(8192)] * 16, "t4", shuffle=True, append=1)
    if name == "long128k":
        return Workload(name, 1, [sc(131072)], "t4", shuffle=True, needle=True)
    if name == "prefill":
        return Workload(name, 4, [0] * 4, "t4", shuffle=True,
                        append=sc(32768))
    if name == "ragged":
        g = torch.Generator().manual_seed(1000 + seed)
        lo, hi = sc(1024), sc(32768)
        ctx = torch.randint(lo, hi + 1, (128,), generator=g).tolist()
        return Workload(name, 128, ctx, "t4", shuffle=True, append=1)
    raise ValueError(f"unknown workload {name!r}")


WORKLOADS = ("tiny", "decode8k", "long128k", "prefill", "ragged")


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def rotations_fp64(h_kv: int, seed: int) -> tuple[torch.Tensor, torch.Tensor]:
    """R_k, R_v float64 [h_kv][128][128] (CPU): sign-fixed QR of seeded
    Gaussian matrices (orthogonal to fp64 rounding)."""
    g = _gen(seed * 7919 + 17, "cpu")
    out = []
    for _ in range(2):
        Rs = []
        for _ in range(h_kv):
            A = torch.randn(D, D, generator=g, dtype=torch.float64)
            Q, Rq = torch.linalg.qr(A)
            Q = Q * torch.sign(torch.diagonal(Rq)).unsqueeze(0)
            Rs.append(Q)
        out.append(torch.stack(Rs))
    return out[0], out[1]


def rotations(h_kv: int, seed: int) -> tuple[torch.Tensor, torch.Tensor]:
    """The matrices of rotations_fp64() cast to float32 (what both the
    library and the oracle consume)."""
    R_k, R_v = rotations_fp64(h_kv, seed)
    return R_k.to(torch.float32), R_v.to(torch.float32)


def _draw(n: int, dist: str, g: torch.Generator, device) -> torch.Tensor:
    """n float32 samples of N(0,1) or Student-t with nu = 4 (a standard normal
    over the root of a chi-square(4)/4 built from four more normals)."""
    out = torch.empty(n, dtype=torch.float32, device=device)
    for s in range(0, n, _CHUNK):
        m = min(_CHUNK, n - s)
        z = torch.randn(m, generator=g, device=device)
        if dist == "t4":
            c = torch.randn(4, m, generator=g, device=device)
            z = z / torch.sqrt((c * c).sum(0) / 4.0)
        elif dist != "normal":
            raise ValueError(dist)
        out[s:s + m] = z
    return out


def key_offsets(h_kv: int, seed: int) -> torch.Tensor:
    """float32 [h_kv][128]: 4 random channels per head get sign * U(6, 10)."""
    g = _gen(seed * 104729 + 3, "cpu")
    off = torch.zeros(h_kv, D)
    for h in range(h_kv):
        ch = torch.randperm(D, generator=g)[:4]
        mag = 6.0 + 4.0 * torch.rand(4, generator=g)
        sign = torch.where(torch.rand(4, generator=g) < 0.5, -1.0, 1.0)
        off[h, ch] = mag * sign
    return off


def kv_tokens(n_tok: int, h_kv: int, dist: str, seed: int, stream: int,
              device="cpu") -> tuple[torch.Tensor, torch.Tensor]:
    """bf16 K, V [n_tok][h_kv][128]; keys carry the per-head offsets.
    ``stream`` separates independent draws (context vs appended tokens)."""
    g = _gen(seed * 1000003 + 11 * stream + 1, device)
    n = n_tok * h_kv * D
    k = _draw(n, dist, g, device).view(n_tok, h_kv, D)
    k += key_offsets(h_kv, seed).to(device).unsqueeze(0)
    v = _draw(n, dist, g, device).view(n_tok, h_kv, D)
    return k.to(torch.bfloat16), v.to(torch.bfloat16)


def key_mean(k: torch.Tensor) -> torch.Tensor:
    """Harness-side mu: float64 per-(head, channel) mean of bf16 keys
    [n][h_kv][128], returned as float32 (CPU)."""
    acc = torch.zeros(k.shape[1], D, dtype=torch.float64, device=k.device)
    for s in range(0, k.shape[0], 1 << 16):
        acc += k[s:s + (1 << 16)].to(torch.float64).sum(0)
    return (acc / max(k.shape[0], 1)).to(torch.float32).cpu()


def queries(B: int, h_q: int, seed: int, device="cpu") -> torch.Tensor:
    g = _gen(seed * 31337 + 5, device)
    return torch.randn(B, h_q, D, generator=g, device=device).to(torch.bfloat16)


def page_tables(seq_tokens: list, shuffle: bool, seed: int):
    """Block table int32 [B][max_pages] (unused entries -1) covering
    seq_tokens[b] positions per sequence, and the physical page count.
    Shuffled tables draw a random permutation of all physical pages, so the
    pages of different sequences interleave."""
    n_pages = [(t + PAGE - 1) // PAGE for t in seq_tokens]
    total = sum(n_pages)
    max_pages = max(max(n_pages), 1)
    if shuffle:
        g = _gen(seed * 65537 + 7, "cpu")
        perm = torch.randperm(total, generator=g).to(torch.int32)
    else:
        perm = torch.arange(total, dtype=torch.int32)
    bt = torch.full((len(seq_tokens), max_pages), -1, dtype=torch.int32)
    o = 0
    for b, n in enumerate(n_pages):
        bt[b, :n] = perm[o:o + n]
        o += n
    return bt, max(total, 1)


def plant_needles(k: torch.Tensor, cu: list, mu: torch.Tensor,
                  q: torch.Tensor, seed: int, cosine: float = 0.9):
    """Replace one context key per KV head of sequence 0 by a needle whose
    centered part (k - mu) has the given cosine with the query of the
    group's first query head and the mean norm of the centered keys.
    Returns the needle positions [h_kv] (positions within sequence 0)."""
    h_kv = k.shape[1]
    ratio = q.shape[1] // h_kv
    n0 = cu[1] - cu[0]
    g = _gen(seed * 271 + 9, "cpu")
    pos = torch.randint(0, n0, (h_kv,), generator=g)
    for h in range(h_kv):
        kc = k[cu[0]:cu[1], h].to(torch.float64) - mu[h].to(k.device, torch.float64)
        norm = kc.norm(dim=1).mean().item()
        qd = q[0, h * ratio].to(torch.float64).cpu()
        u = qd / qd.norm()
        w = torch.randn(D, generator=g, dtype=torch.float64)
        w = w - (w @ u) * u
        w = w / w.norm()
        vec = norm * (cosine * u + (1.0 - cosine ** 2) ** 0.5 * w)
        val = (mu[h].to(torch.float64) + vec).to(torch.bfloat16)
        k[cu[0] + int(pos[h]), h] = val.to(k.device)
    return pos


def build_case(wl: Workload, seed: int = 0, device="cpu") -> dict:
    """Every tensor of one workload.  Context tokens are those to prefill the
    cache with (``k_ctx``/``v_ctx``, rows grouped by sequence per
    ``cu_ctx``); the step appends ``k_new``/``v_new`` (``append`` per
    sequence) at positions ctx[b].. and then decodes over ctx[b] + append."""
    B, h_q, h_kv = wl.B, wl.h_q, wl.h_kv
    R_k, R_v = rotations(h_kv, seed)
    ctx = list(wl.ctx)
    cu_ctx = [0]
    for c in ctx:
        cu_ctx.append(cu_ctx[-1] + c)
    k_ctx, v_ctx = kv_tokens(cu_ctx[-1], h_kv, wl.dist, seed, 0, device)
    n_new = wl.append * B
    k_new, v_new = kv_tokens(n_new, h_kv, wl.dist, seed, 1, device)
    allk = torch.cat([k_ctx, k_new]) if n_new else k_ctx
    mu = key_mean(allk) if allk.shape[0] else torch.zeros(h_kv, D)
    q = queries(B, h_q, seed, device)
    needle = None
    if wl.needle:
        needle = plant_needles(k_ctx, cu_ctx, mu, q, seed)
    total = [c + wl.append for c in ctx]
    bt, num_pages = page_tables(total, wl.shuffle, seed)
    cu_new = [b * wl.append for b in range(B + 1)]
    return dict(
        R_k=R_k, R_v=R_v, mu=mu, q=q,
        k_ctx=k_ctx, v_ctx=v_ctx,
        cu_ctx=torch.tensor(cu_ctx, dtype=torch.int32),
        pos0_ctx=torch.zeros(B, dtype=torch.int32),
        k_new=k_new, v_new=v_new,
        cu_new=torch.tensor(cu_new, dtype=torch.int32),
        pos0_new=torch.tensor(ctx, dtype=torch.int32),
        seq_lens=torch.tensor(total, dtype=torch.int32),
        seq_lens_ctx=torch.tensor(ctx, dtype=torch.int32),
        block_table=bt, num_pages=num_pages, needle=needle,
        h_q=h_q, h_kv=h_kv, B=B)


def bf16_bits(t: torch.Tensor):
    """Raw uint16 bit patterns of a bf16 tensor as a numpy array (CPU)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view("uint16")


def calib_trace(seed: int, T: int, nt: int, g: int = 4, d_model: int = 64,
                device="cpu"):
    """A synthetic calibration trace of one KV head, float64 (stands in for
    the paper's BF16 GPQA Q/K/V traces): keys Student-t(4) with the 4
    offset channels of key_offsets() (head 0 of ``seed``), values
    Student-t(4), the g query heads ~ N(0, 1) at the last nt positions, and
    a random output projection W_O [g][d_model][128] ~ N(0, 1/(g*128)).
    Returns q [nt][g][128], K, V [T][128], W_O, t_pos int32 [nt]."""
    gen = _gen(seed * 7919 + 17, "cpu")
    K = _draw(T * D, "t4", gen, "cpu").view(T, D).to(torch.float64)
    K += key_offsets(1, seed)[0].to(torch.float64)
    V = _draw(T * D, "t4", gen, "cpu").view(T, D).to(torch.float64)
    q = torch.randn(nt, g, D, generator=gen, dtype=torch.float64)
    W_O = torch.randn(g, d_model, D, generator=gen, dtype=torch.float64) / math.sqrt(g * D)
    t_pos = torch.arange(T - nt, T, dtype=torch.int32)
    return (q.to(device), K.to(device), V.to(device), W_O.to(device),
            t_pos.to(device))
