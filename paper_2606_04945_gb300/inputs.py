"""Seeded synthetic inputs shaped like the paper's DLLM workloads.

This module is shared by the tests, the bench and the smoke check: it feeds
the same arrays to the CUDA path and to the CPU oracle. It holds no
arithmetic of the method (no transform, quantiser, GEMM or TAC): only random
draws and the synthetic stand-ins for calibrated parameters (per-state
smoothing scales, TAC blocks). No model weights, calibration set or benchmark
items are used; the paper evaluates LLaDA-8B and Dream-7B (Sec. 4.1) and these
arrays stand in for their activations and weights.

Arrays are numpy: activations and weights in float16 (bfloat16 workloads are
returned as float32 values already rounded to bfloat16, plus a dtype tag),
masks as uint8 (1 = masked), scales and TAC parameters as float32.
"""

from dataclasses import dataclass, field
from typing import Optional

import numpy as np


def round_to_bf16(x):
    """float32 values rounded to the nearest bfloat16 (ties to even), kept in
    float32 storage (numpy has no bfloat16 dtype)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    u = (u + 0x7FFF + lsb) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


@dataclass
class SgatParams:
    """The two state transforms of one linear and its shared weight transform.

    a_m / a_u: per-state diagonal smoothing applied before the Hadamard
    block hb; inv_a_w: the weight-side inverse smoothing; (d_sh, d_m, d_u):
    the gate layout over transformed coordinates.
    """
    K: int
    hb: int
    a_m: np.ndarray
    a_u: np.ndarray
    inv_a_w: np.ndarray
    d_sh: int
    d_m: int
    d_u: int


@dataclass
class TacParams:
    C: int
    g: int
    M: np.ndarray  # float32 [C/g, g, g]
    d: np.ndarray  # float32 [C/g, g]


@dataclass
class LinearCase:
    """One SGAT linear: Y = SGAT-W4A4(X) with optional TAC on its input."""
    name: str
    X: np.ndarray            # [L, K] float16, or float32 holding bf16 values
    dtype: str               # "f16" or "bf16": element type of X, W and Y
    mask: np.ndarray         # [L] uint8
    W: np.ndarray            # [N, K] same storage rule as X
    xf: SgatParams
    bias: Optional[np.ndarray] = None   # [N] float32
    tac: Optional[TacParams] = None
    meta: dict = field(default_factory=dict)

    @property
    def L(self):
        return self.X.shape[0]

    @property
    def K(self):
        return self.X.shape[1]

    @property
    def N(self):
        return self.W.shape[0]


def hadamard_block(K, cap=4096):
    """Largest power of two dividing K, capped (512 -> 512, 4096 -> 4096,
    12288 -> 4096, 3584 -> 512, 18944 -> 512)."""
    hb = 1
    while K % (hb * 2) == 0 and hb * 2 <= cap:
        hb *= 2
    return hb


def smoothing_scales(X, mask):
    """Synthetic calibration of the per-state diagonal smoothing: for state s,
    a_s[j] = (max_{i in I_s} |X[i, j]|)^(-1/2), renormalised to geometric mean
    one (SmoothQuant-style migration strength 0.5 with no weight term).
    The weight side uses a_w = sqrt(a_m * a_u). A state with no tokens gets
    ones. Returns (a_m, a_u, inv_a_w) as float32."""
    X = np.abs(np.asarray(X, dtype=np.float32))
    K = X.shape[1]
    out = []
    for state in (1, 0):
        rows = X[np.asarray(mask) == state]
        if rows.shape[0] == 0:
            out.append(np.ones(K, np.float64))
            continue
        mx = np.maximum(rows.max(axis=0).astype(np.float64), 1e-3)
        a = mx ** -0.5
        a = a / np.exp(np.mean(np.log(a)))
        out.append(a)
    a_m, a_u = out
    a_w = np.sqrt(a_m * a_u)
    return (a_m.astype(np.float32), a_u.astype(np.float32), (1.0 / a_w).astype(np.float32))


def default_gates(K, on=True):
    """d_m = d_u = K / 32 with the rest shared (App. B), or all-shared."""
    if not on:
        return K, 0, 0
    d_m = d_u = K // 32
    return K - d_m - d_u, d_m, d_u


def make_sgat(X, mask, gates_on=True, hb=None):
    K = X.shape[1]
    a_m, a_u, inv_a_w = smoothing_scales(X, mask)
    d_sh, d_m, d_u = default_gates(K, gates_on)
    return SgatParams(K=K, hb=hb or hadamard_block(K), a_m=a_m, a_u=a_u,
                      inv_a_w=inv_a_w, d_sh=d_sh, d_m=d_m, d_u=d_u)


def make_tac(rng, C, g, noise=0.01):
    B = C // g
    M = np.eye(g, dtype=np.float32)[None] + rng.normal(0, noise, (B, g, g)).astype(np.float32)
    d = rng.normal(0, noise, (B, g)).astype(np.float32)
    return TacParams(C=C, g=g, M=M.astype(np.float32), d=d)


def _store(x, dtype):
    return x.astype(np.float16) if dtype == "f16" else round_to_bf16(x)


def heavy_tail_activations(rng, L, K, frac=0.005, nu=3.0, dtype="f16"):
    """N(0, 1) activations with a fraction of channels drawn Student-t(nu)."""
    X = rng.standard_normal((L, K), dtype=np.float32)
    n_heavy = max(1, int(round(frac * K)))
    cols = rng.choice(K, n_heavy, replace=False)
    X[:, cols] = rng.standard_t(nu, (L, n_heavy)).astype(np.float32)
    return _store(X, dtype)


def outlier_activations(rng, L, K, mask, n_out=8, scale_u=20.0, scale_m=5.0, dtype="f16"):
    """N(0, 1) activations with n_out outlier channels scaled by scale_u on
    unmasked tokens and scale_m on masked tokens."""
    X = rng.standard_normal((L, K), dtype=np.float32)
    cols = rng.choice(K, n_out, replace=False)
    mult = np.where(np.asarray(mask)[:, None] == 1, scale_m, scale_u).astype(np.float32)
    X[:, cols] *= mult
    return _store(X, dtype)


def gaussian_weight(rng, N, K, std=0.02, dtype="f16"):
    return _store(rng.normal(0, std, (N, K)).astype(np.float32), dtype)


# ---------------------------------------------------------------------------
# Workloads
# ---------------------------------------------------------------------------

def single_linear(seed=0, gates_on=True):
    """Single SGAT linear, 256 tokens x K=512 -> N=512: Bernoulli(0.5) mask,
    8 outlier channels (x20 unmasked, x5 masked), W ~ N(0, 0.02), one
    512-point Hadamard; TAC with block 64 and blocks I + N(0, 0.01)."""
    rng = np.random.default_rng(seed)
    L, K, N = 256, 512, 512
    mask = (rng.random(L) < 0.5).astype(np.uint8)
    X = outlier_activations(rng, L, K, mask)
    W = gaussian_weight(rng, N, K)
    xf = make_sgat(X, mask, gates_on=gates_on, hb=512)
    tac = make_tac(rng, K, 64)
    return LinearCase("single_linear_256x512x512", X, "f16", mask, W, xf, tac=tac,
                      meta=dict(seed=seed, gates_on=gates_on))


def llada_attention_mask(L=1024, prompt=512, masked_frac=0.75):
    """Prompt positions unmasked; generated positions unmasked except a
    masked suffix covering masked_frac of them (0..639 unmasked, 640..1023
    masked at the defaults)."""
    gen = L - prompt
    n_masked = int(round(masked_frac * gen))
    mask = np.zeros(L, np.uint8)
    mask[L - n_masked:] = 1
    return mask


def llada_attention(seed=0):
    """LLaDA-8B attention projections at one denoising step: 1024 tokens,
    hidden 4096, fused QKV 4096 -> 12288 and O 4096 -> 4096, FP16 inputs with
    0.5% Student-t(3) channels, TAC on the attention output with 128 x 128
    per-head blocks (32 heads). Returns (qkv LinearCase, o LinearCase)."""
    rng = np.random.default_rng(seed)
    L, H = 1024, 4096
    mask = llada_attention_mask(L)
    X = heavy_tail_activations(rng, L, H)
    W_qkv = gaussian_weight(rng, 3 * H, H)
    qkv = LinearCase("llada_qkv_1024x4096x12288", X, "f16", mask, W_qkv, make_sgat(X, mask))
    Z = heavy_tail_activations(rng, L, H)
    W_o = gaussian_weight(rng, H, H)
    tac = make_tac(rng, H, 128)
    o = LinearCase("llada_o_1024x4096x4096", Z, "f16", mask, W_o, make_sgat(Z, mask), tac=tac)
    return qkv, o


def semi_ar_mask(L=1024, block=32, ratio=0.5):
    """The last round(ratio * L/block) of the L/block contiguous blocks are
    masked (semi-autoregressive block decoding)."""
    nb = L // block
    n_masked = int(round(ratio * nb))
    mask = np.zeros(L, np.uint8)
    if n_masked:
        mask[L - n_masked * block:] = 1
    return mask


def llada_mlp(seed=0, ratio=0.5):
    """LLaDA-8B MLP at one step: 1024 tokens, gate+up 4096 -> 2 x 12288,
    SwiGLU, down 12288 -> 4096. Returns (gate_up LinearCase, W_down, mask,
    down-input generator rng). The down projection's input is the SwiGLU of
    the gate/up output, so its case is built by the caller from that."""
    rng = np.random.default_rng(seed + 1000 * int(round(ratio * 10)))
    L, H, F = 1024, 4096, 12288
    mask = semi_ar_mask(L, 32, ratio)
    X = heavy_tail_activations(rng, L, H)
    W_gu = gaussian_weight(rng, 2 * F, H)
    gu = LinearCase(f"llada_gate_up_1024x4096x24576_r{ratio}", X, "f16", mask, W_gu,
                    make_sgat(X, mask), meta=dict(ratio=ratio))
    W_down = gaussian_weight(rng, H, F)
    return gu, W_down, mask


def remask_schedule(rng, S, gen_len, still_masked):
    """Low-confidence remasking at a mid-trajectory step: of the last gen_len
    positions, the still_masked ones with the lowest seeded confidence stay
    masked; the prompt is unmasked."""
    mask = np.zeros(S, np.uint8)
    conf = rng.random(gen_len)
    order = np.argsort(conf)
    mask[S - gen_len + order[:still_masked]] = 1
    return mask


def dream_block_linears(seed=0, batch=4, seq=2048, gen_len=256):
    """Dream-7B (Qwen2.5-7B shape) block linears on 4 x 2048 = 8192 tokens in
    bfloat16: QKV 3584 -> 4608 with bias, O 3584 -> 3584 with TAC (block 128
    per head), gate+up 3584 -> 2 x 18944, down 18944 -> 3584. Mask: per
    sequence, 128 of the last 256 positions still masked by seeded
    low-confidence remasking."""
    rng = np.random.default_rng(seed)
    H, F, nq, nkv, dh = 3584, 18944, 28, 4, 128
    L = batch * seq
    mask = np.concatenate([remask_schedule(rng, seq, gen_len, gen_len // 2) for _ in range(batch)])
    cases = []
    X = heavy_tail_activations(rng, L, H, dtype="bf16")
    Wqkv = gaussian_weight(rng, (nq + 2 * nkv) * dh, H, dtype="bf16")
    bias = rng.normal(0, 0.02, (nq + 2 * nkv) * dh).astype(np.float32)
    cases.append(LinearCase("dream_qkv_8192x3584x4608", X, "bf16", mask, Wqkv, make_sgat(X, mask), bias=bias))
    Z = heavy_tail_activations(rng, L, H, dtype="bf16")
    Wo = gaussian_weight(rng, H, H, dtype="bf16")
    cases.append(LinearCase("dream_o_8192x3584x3584", Z, "bf16", mask, Wo, make_sgat(Z, mask),
                            tac=make_tac(rng, H, 128)))
    X2 = heavy_tail_activations(rng, L, H, dtype="bf16")
    Wgu = gaussian_weight(rng, 2 * F, H, dtype="bf16")
    cases.append(LinearCase("dream_gate_up_8192x3584x37888", X2, "bf16", mask, Wgu, make_sgat(X2, mask)))
    X3 = heavy_tail_activations(rng, L, F, dtype="bf16")
    Wd = gaussian_weight(rng, H, F, dtype="bf16")
    cases.append(LinearCase("dream_down_8192x18944x3584", X3, "bf16", mask, Wd, make_sgat(X3, mask)))
    return cases


@dataclass
class DreamBlockCase:
    """One Dream-7B (Qwen2.5-7B shape) transformer block at a denoising step:
    the input hidden states, the mask, the token positions, the block's
    random-init bf16 weights and the synthetic stand-ins for its calibrated
    parameters (per-linear SGAT transforms, TAC blocks per head)."""
    X: np.ndarray            # [L, hidden] float32 holding bf16 values
    mask: np.ndarray         # [L] uint8
    pos: np.ndarray          # [L] int32, position within the sequence
    batch: int
    seq: int
    hidden: int
    ffn: int
    heads: int
    kv_heads: int
    w_ln1: np.ndarray        # [hidden] float32 RMSNorm gains
    w_ln2: np.ndarray
    W_qkv: np.ndarray        # [(heads + 2 kv_heads) 128, hidden] bf16 values
    b_qkv: np.ndarray        # float32 bias
    W_o: np.ndarray          # [hidden, hidden]
    W_gate: np.ndarray       # [ffn, hidden]
    W_up: np.ndarray         # [ffn, hidden]
    W_down: np.ndarray       # [hidden, ffn]
    tac: TacParams           # one 128 x 128 block per query head
    xf_qkv: SgatParams
    xf_o: SgatParams
    xf_gu: SgatParams
    xf_down: SgatParams
    rope_theta: float = 1e6
    eps: float = 1e-6

    @property
    def L(self):
        return self.X.shape[0]


def dream_block(seed=0, batch=4, seq=2048, gen_len=256, hidden=3584, ffn=18944, heads=28, kv_heads=4):
    """The Dream-7B block workload: 4 sequences of 2048 tokens in bfloat16,
    the last 256 positions of each generated with 128 still masked
    (seeded low-confidence remasking). Weights N(0, 0.02), RMSNorm gains
    1 + N(0, 0.1), QKV bias N(0, 0.02), TAC blocks I + N(0, 0.01) per head.
    The per-state smoothing of every linear is the synthetic calibration on
    heavy-tailed activations of that linear's width (the block input itself
    for the QKV projection); rows of 2048 tokens with the block's mask
    pattern stand in for the calibration set."""
    rng = np.random.default_rng(seed)
    L = batch * seq
    mask = np.concatenate([remask_schedule(rng, seq, gen_len, gen_len // 2) for _ in range(batch)])
    pos = np.tile(np.arange(seq, dtype=np.int32), batch)
    X = heavy_tail_activations(rng, L, hidden, dtype="bf16")
    nqkv = (heads + 2 * kv_heads) * 128
    g = lambda n, k: gaussian_weight(rng, n, k, dtype="bf16")
    W_qkv, W_o, W_gate, W_up, W_down = g(nqkv, hidden), g(hidden, hidden), g(ffn, hidden), g(ffn, hidden), g(hidden, ffn)
    b_qkv = rng.normal(0, 0.02, nqkv).astype(np.float32)
    w_ln1 = (1.0 + rng.normal(0, 0.1, hidden)).astype(np.float32)
    w_ln2 = (1.0 + rng.normal(0, 0.1, hidden)).astype(np.float32)
    tac = make_tac(rng, hidden, 128)
    calib_mask = mask[:seq]
    calib = lambda K: make_sgat(heavy_tail_activations(rng, seq, K, dtype="bf16"), calib_mask)
    return DreamBlockCase(X=X, mask=mask, pos=pos, batch=batch, seq=seq, hidden=hidden, ffn=ffn, heads=heads,
                          kv_heads=kv_heads, w_ln1=w_ln1, w_ln2=w_ln2, W_qkv=W_qkv, b_qkv=b_qkv, W_o=W_o,
                          W_gate=W_gate, W_up=W_up, W_down=W_down, tac=tac, xf_qkv=make_sgat(X, mask),
                          xf_o=calib(hidden), xf_gu=calib(hidden), xf_down=calib(ffn))


def basis_calibration_set(seed, d, n_samples=16, tokens=64, N=None, mask_p=0.5):
    """Synthetic calibration set for the dense basis (App. B): n_samples
    activation matrices of `tokens` tokens each (one per denoising step,
    N(0, 1) with 0.5% Student-t(3) channels, float32), each with its own
    Bernoulli(mask_p) mask, and a weight N(0, 0.02) [N][d] (N = d by
    default). Returns (samples [(X, mask)], W)."""
    rng = np.random.default_rng(seed)
    samples = []
    for _ in range(n_samples):
        mask = (rng.random(tokens) < mask_p).astype(np.uint8)
        X = heavy_tail_activations(rng, tokens, d, dtype="f16").astype(np.float32)
        samples.append((X, mask))
    W = gaussian_weight(rng, N or d, d).astype(np.float32)
    return samples, W


def random_linear(seed, L, K, N, dtype="f16", gates_on=True, tac_g=None, bias=False,
                  mask_p=0.5, hb=None):
    """Small random case for shape sweeps (ragged L, several tiles)."""
    rng = np.random.default_rng(seed)
    mask = (rng.random(L) < mask_p).astype(np.uint8)
    X = outlier_activations(rng, L, K, mask, n_out=min(8, K // 16), dtype=dtype)
    W = gaussian_weight(rng, N, K, dtype=dtype)
    xf = make_sgat(X, mask, gates_on=gates_on, hb=hb)
    b = rng.normal(0, 0.02, N).astype(np.float32) if bias else None
    tac = make_tac(rng, K, tac_g) if tac_g else None
    return LinearCase(f"random_{L}x{K}x{N}", X, dtype, mask, W, xf, bias=b, tac=tac)


def tac_calibration_pairs(seed, N, C, g, dtype="f16"):
    """Paired calibration outputs for TAC (App. C): Z_fp [N][C] with
    correlated channels inside each g-block (Gaussian tokens through a
    random g x g mixing near I) and per-channel means, and Z_q = Z_fp plus
    per-token noise as wide as a 4-bit step (uniform over one step of
    amax / 7, the width of a 4-bit quantiser's rounding error) and a small
    Gaussian term. Both are rounded to `dtype` (float16 arrays, or bfloat16
    values held in float32)."""
    rng = np.random.default_rng(seed)
    B = C // g
    mix = rng.standard_normal((B, g, g)) / np.sqrt(g) + np.eye(g)[None]
    Z = np.einsum("nbi,bij->nbj", rng.standard_normal((N, B, g)), mix).reshape(N, C)
    Z = Z + rng.normal(0.0, 0.5, C)[None, :]
    step = np.abs(Z).max(axis=1, keepdims=True) / 7.0
    Zq = Z + step * rng.uniform(-0.5, 0.5, Z.shape) + rng.normal(0.0, 0.01, Z.shape)
    return _store(Z, dtype), _store(Zq, dtype)
