"""Oracle: SGAT transform, symmetric quantisers, integer GEMM, dequantisation.

Test infrastructure only (see the package docstring): the CUDA path never
imports this module.

Notation follows the paper. ``X`` is the input activation (L x d, written K
here for the reduction length), ``W`` the weight (C x d, written N x K),
``mask`` the per-token state (1 = masked ``m``, 0 = unmasked ``u``), ``P`` the
transformation basis, ``G_m`` / ``G_u`` the binary subspace gates.

Readings of the paper taken here:

* The quantiser is the symmetric signed member of the uniform family of
  Eq. 2-3: zero point 0, codes in [-qmax, qmax] with qmax = 2^(b-1) - 1.
  ``round`` is round-half-to-even. The scale form is s = amax / qmax and the
  code is rne(v * r) with r = qmax / amax, both in float32. An all-zero row
  gets s = 0 and all-zero codes.
* The asymmetric member (Eq. 2-4), for activations: per row, X_min and
  X_max are the row's extremes with zero included (X_min <= 0 <= X_max, so
  z stays in [0, 2^b - 1]); s = fl(fl(X_max - X_min) / (2^b - 1)); X / s is
  taken as fl(v * r) with r = fl((2^b - 1) / fl(X_max - X_min)), like the
  symmetric reading; z = rne(fl(-X_min * r)); codes clamp(rne(fl(v r)) + z,
  0, 2^b - 1). An all-zero row gets s = 0, z = 0 and all-zero codes.
* The dense basis (SGAT's learned P, kept orthogonal, App. B: W_f =
  Q_w(P^T W^T)): the transform is a 16-bit GEMM. Its operands are the
  scaled rows fl32(x * a_s) and P, both rounded to float16; the product is
  exact here (float64) and rounded to float16 once (the stored result),
  then gated and quantised. The weight side is the same product on
  fl32(w * inv_a_w): w_f = fl16(fl16(w * inv_a_w) P), the row form of
  P^T W^T.
* P is the block-diagonal Sylvester Hadamard matrix of block ``hb`` preceded
  by a per-state diagonal smoothing ``a_s``: Phi_s(x) = ((x * a_s) H) G_s with
  the unnormalised H; the 1/hb that makes H^-1 = H / hb is folded into the
  weight side (Eq. 12 with P_e = P^-1).
* The subspaces of Eq. 8 occupy transformed coordinates in the order
  [shared | masked-specific | unmasked-specific].
* The Hadamard product x @ H is taken by the fast Walsh-Hadamard transform:
  stages h = 1, 2, 4, ..., hb/2, each butterfly (a, b) -> (a + b, a - b)
  rounded to float32.
"""

import numpy as np

F32 = np.float32


# ---------------------------------------------------------------------------
# Basis (Eq. 8, Hadamard reading) and gates (Eq. 9)
# ---------------------------------------------------------------------------

def hadamard_sylvester(n):
    """Dense Sylvester Hadamard matrix H_n (int64), H_2n = [[H, H], [H, -H]].

    Used by the pins only; the transform itself runs the fast algorithm.
    """
    assert n >= 1 and (n & (n - 1)) == 0, "Sylvester order must be a power of 2"
    H = np.ones((1, 1), dtype=np.int64)
    while H.shape[0] < n:
        H = np.block([[H, H], [H, -H]])
    return H


def state_gates(K, d_sh, d_m, d_u):
    """Binary subspace gates of Eq. 9 as 0/1 float32 vectors (g_m, g_u).

    G_m = diag(1_{d_sh}, 1_{d_m}, 0_{d_u}) and G_u = diag(1_{d_sh}, 0_{d_m},
    1_{d_u}) with d = d_sh + d_m + d_u (Eq. 8).
    """
    assert d_sh >= 0 and d_m >= 0 and d_u >= 0 and d_sh + d_m + d_u == K
    g_m = np.zeros(K, dtype=F32)
    g_u = np.zeros(K, dtype=F32)
    g_m[:d_sh] = 1
    g_u[:d_sh] = 1
    g_m[d_sh:d_sh + d_m] = 1
    g_u[d_sh + d_m:] = 1
    return g_m, g_u


def fwht_f32(x, hb):
    """x @ H_hb on every hb-block of the last axis, in float32.

    The fast Walsh-Hadamard transform: for h = 1, 2, 4, ..., hb/2, every pair
    (j, j + h) inside each aligned 2h-block is replaced by
    (x_j + x_{j+h}, x_j - x_{j+h}), each result rounded to float32.
    """
    x = np.array(x, dtype=F32, copy=True)
    K = x.shape[-1]
    assert hb >= 1 and (hb & (hb - 1)) == 0 and K % hb == 0
    lead = x.shape[:-1]
    h = 1
    while h < hb:
        y = x.reshape(*lead, K // (2 * h), 2, h)
        a = y[..., 0, :].copy()
        b = y[..., 1, :].copy()
        y[..., 0, :] = a + b
        y[..., 1, :] = a - b
        x = y.reshape(*lead, K)
        h *= 2
    return x


# ---------------------------------------------------------------------------
# Quantisers (Eq. 2-3, symmetric reading) and int4 packing
# ---------------------------------------------------------------------------

def qmax_of(bits):
    assert 2 <= bits <= 16
    return (1 << (bits - 1)) - 1


def quantize_rows_sym(v, bits):
    """Per-row symmetric quantiser (Eq. 2 with z = 0, Sec. 3.1 granularity).

    Returns (codes int32 [rows, K], s float32 [rows]). Rows are tokens for
    Q_a (per-token) and output channels for Q_w (per-channel).
    """
    v = np.asarray(v, dtype=F32)
    assert v.ndim == 2
    assert np.all(np.isfinite(v)), "the quantiser is defined on finite inputs"
    qmax = F32(qmax_of(bits))
    amax = np.max(np.abs(v), axis=1) if v.shape[1] else np.zeros(v.shape[0], F32)
    nz = amax > 0
    safe = np.where(nz, amax, F32(1))
    s = np.where(nz, safe / qmax, F32(0)).astype(F32)
    r = np.where(nz, qmax / safe, F32(0)).astype(F32)
    prod = (v * r[:, None]).astype(F32)
    q = np.clip(np.rint(prod), -qmax, qmax).astype(np.int32)
    return q, s


def quantize_rows_asym(v, bits):
    """Per-row asymmetric quantiser (Eq. 2-4, read as in the module notes).

    Returns (codes int32 [rows, K] in [0, 2^b - 1], s float32 [rows],
    z int32 [rows]); X_hat = s (codes - z) (Eq. 3).
    """
    v = np.asarray(v, dtype=F32)
    assert v.ndim == 2
    assert np.all(np.isfinite(v)), "the quantiser is defined on finite inputs"
    levels = F32((1 << bits) - 1)
    vmax = np.maximum(v.max(axis=1), F32(0)) if v.shape[1] else np.zeros(v.shape[0], F32)
    vmin = np.minimum(v.min(axis=1), F32(0)) if v.shape[1] else np.zeros(v.shape[0], F32)
    d = (vmax - vmin).astype(F32)
    nz = d > 0
    safe = np.where(nz, d, F32(1))
    s = np.where(nz, safe / levels, F32(0)).astype(F32)
    r = np.where(nz, levels / safe, F32(0)).astype(F32)
    z = np.clip(np.rint((-vmin * r).astype(F32)), 0, levels).astype(np.int32)
    prod = (v * r[:, None]).astype(F32)
    q = np.clip(np.rint(prod) + z[:, None], 0, levels).astype(np.int32)
    return q, s, z


def pack_int4(q):
    """Pack int4 codes [rows, K] into bytes [rows, K/2].

    Code k goes to byte k // 2; even k in the low nibble, odd k in the high
    nibble; each nibble holds the code in two's complement.
    """
    q = np.asarray(q)
    assert q.shape[-1] % 2 == 0
    assert q.min(initial=0) >= -8 and q.max(initial=0) <= 7
    u = (q.astype(np.int64) & 0xF).astype(np.uint8)
    return (u[..., 0::2] | (u[..., 1::2] << 4)).astype(np.uint8)


def unpack_int4(p):
    """Inverse of ``pack_int4``: bytes [rows, K/2] -> int32 codes [rows, K]."""
    p = np.asarray(p, dtype=np.uint8)
    lo = (p & 0xF).astype(np.int32)
    hi = (p >> 4).astype(np.int32)
    lo = np.where(lo >= 8, lo - 16, lo)
    hi = np.where(hi >= 8, hi - 16, hi)
    out = np.empty(p.shape[:-1] + (2 * p.shape[-1],), dtype=np.int32)
    out[..., 0::2] = lo
    out[..., 1::2] = hi
    return out


# ---------------------------------------------------------------------------
# Weight side (Eq. 12, App. B folding)
# ---------------------------------------------------------------------------

def transform_weight_f32(W, inv_a_w, hb):
    """Unquantised folded weight rows: ((W[n] * inv_a_w) H_hb) / hb, float32.

    Row n of the result is column n of P_e W^T with P_e = P^-1 for the basis
    P = diag(a_w) H: P^-1 = H diag(1 / a_w) / hb (H is symmetric).
    """
    w = np.asarray(W).astype(F32)
    if inv_a_w is not None:
        w = (w * np.asarray(inv_a_w, dtype=F32)[None, :]).astype(F32)
    t = fwht_f32(w, hb)
    return (t * F32(1.0 / hb)).astype(F32)


def prepare_weight(W, inv_a_w, hb, bits):
    """W_f = Q_w(P_e W^T) (Eq. 12, App. B), per-output-channel symmetric.

    Returns (codes int32 [N, K], s_w float32 [N]).
    """
    return quantize_rows_sym(transform_weight_f32(W, inv_a_w, hb), bits)


# ---------------------------------------------------------------------------
# Activation side (Eq. 7, 10, 11, 13): literal state split and scatter
# ---------------------------------------------------------------------------

def state_index_sets(mask):
    """I_m and I_u of Eq. 7 (mask bit 1 = masked)."""
    mask = np.asarray(mask).astype(np.uint8)
    return np.nonzero(mask == 1)[0], np.nonzero(mask == 0)[0]


def phi_state(Xs, a_s, g_s, hb):
    """Phi_s(X^s) = X^s P G_s (Eq. 11) for one state group, float32.

    X^s P = (X^s * a_s) H_hb (one float32 product per element, then the fast
    transform); the gate keeps the shared and own-state coordinates.
    """
    x = np.asarray(Xs).astype(F32)
    if a_s is not None:
        x = (x * np.asarray(a_s, dtype=F32)[None, :]).astype(F32)
    v = fwht_f32(x, hb)
    return np.where(np.asarray(g_s)[None, :] != 0, v, F32(0)).astype(F32)


def sgat_quantize_act(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, bits):
    """Q_a(Phi_s(X^s)) for both states, scattered back to token order.

    Eq. 7 splits tokens by state, Eq. 11 transforms each group with its own
    gate, Q_a quantises per token, and the groups return to their original
    positions. Returns (codes int32 [L, K], s_a float32 [L]).
    """
    X = np.asarray(X)
    L, K = X.shape
    g_m, g_u = state_gates(K, d_sh, d_m, d_u)
    I_m, I_u = state_index_sets(mask)
    codes = np.zeros((L, K), dtype=np.int32)
    s_a = np.zeros(L, dtype=F32)
    for I, a, g in ((I_m, a_m, g_m), (I_u, a_u, g_u)):
        if len(I) == 0:
            continue
        q, s = quantize_rows_sym(phi_state(X[I], a, g, hb), bits)
        codes[I] = q
        s_a[I] = s
    return codes, s_a


def sgat_quantize_act_asym(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, bits=4):
    """As sgat_quantize_act with the asymmetric activation quantiser.
    Returns (codes int32 [L, K] in [0, 2^b - 1], s_a float32 [L], z_a int32
    [L])."""
    X = np.asarray(X)
    L, K = X.shape
    g_m, g_u = state_gates(K, d_sh, d_m, d_u)
    I_m, I_u = state_index_sets(mask)
    codes = np.zeros((L, K), dtype=np.int32)
    s_a = np.zeros(L, dtype=F32)
    z_a = np.zeros(L, dtype=np.int32)
    for I, a, g in ((I_m, a_m, g_m), (I_u, a_u, g_u)):
        if len(I) == 0:
            continue
        q, s, z = quantize_rows_asym(phi_state(X[I], a, g, hb), bits)
        codes[I], s_a[I], z_a[I] = q, s, z
    return codes, s_a, z_a


def dense_basis_product(A, P16):
    """fl16(fl16(A) P) for rows A [rows][K] (float32) and the dense basis P
    [K][K] (float16 values): float64 product of the float16 operands, one
    rounding to float16. Returned as float32."""
    a16 = np.asarray(A, dtype=F32).astype(np.float16).astype(np.float64)
    p = np.asarray(P16, dtype=np.float16).astype(np.float64)
    return (a16 @ p).astype(np.float16).astype(F32)


def sgat_quantize_act_dense(X, mask, a_m, a_u, P16, d_sh, d_m, d_u, bits=4):
    """Q_a(X^s P G_s) with the dense basis (per state: scaled rows, the 16-bit
    product, the gate, the symmetric quantiser). Returns (codes int32 [L, K],
    s_a float32 [L], V float32 [L, K] = the ungated product)."""
    X = np.asarray(X)
    L, K = X.shape
    g_m, g_u = state_gates(K, d_sh, d_m, d_u)
    I_m, I_u = state_index_sets(mask)
    codes = np.zeros((L, K), dtype=np.int32)
    s_a = np.zeros(L, dtype=F32)
    V = np.zeros((L, K), dtype=F32)
    for I, a, g in ((I_m, a_m, g_m), (I_u, a_u, g_u)):
        if len(I) == 0:
            continue
        x = np.asarray(X[I]).astype(F32)
        if a is not None:
            x = (x * np.asarray(a, dtype=F32)[None, :]).astype(F32)
        v = dense_basis_product(x, P16)
        V[I] = v
        q, s = quantize_rows_sym(np.where(np.asarray(g)[None, :] != 0, v, F32(0)).astype(F32), bits)
        codes[I], s_a[I] = q, s
    return codes, s_a, V


def prepare_weight_dense(W, inv_a_w, P16, bits=4):
    """W_f = Q_w(P^T W^T) in row form: rows fl16(fl16(w * inv_a_w) P),
    per-channel symmetric. Returns (codes int32 [N, K], s_w float32 [N],
    Wf float32 [N, K])."""
    w = np.asarray(W).astype(F32)
    if inv_a_w is not None:
        w = (w * np.asarray(inv_a_w, dtype=F32)[None, :]).astype(F32)
    wf = dense_basis_product(w, P16)
    q, s = quantize_rows_sym(wf, bits)
    return q, s, wf


def sgat_transform(X, mask, a_m, a_u, hb, d_sh, d_m, d_u):
    """Phi_s(X^s) for both states in token order, float32, unquantised."""
    X = np.asarray(X)
    L, K = X.shape
    g_m, g_u = state_gates(K, d_sh, d_m, d_u)
    I_m, I_u = state_index_sets(mask)
    V = np.zeros((L, K), dtype=F32)
    for I, a, g in ((I_m, a_m, g_m), (I_u, a_u, g_u)):
        if len(I):
            V[I] = phi_state(X[I], a, g, hb)
    return V


# ---------------------------------------------------------------------------
# Integer GEMM (Eq. 5, Eq. 13) and dequantisation (Eq. 3)
# ---------------------------------------------------------------------------

def int_gemm(qa, qw):
    """acc[i, n] = sum_k qa[i, k] * qw[n, k], exact, returned as int64.

    The products run through a float64 matmul on integer values: every
    partial sum is an integer of magnitude <= K * qmax^2 < 2^53, so the sum is
    exact in any order.
    """
    qa = np.asarray(qa)
    qw = np.asarray(qw)
    assert qa.shape[1] == qw.shape[1]
    bound = qa.shape[1] * int(np.abs(qa).max(initial=0)) * int(np.abs(qw).max(initial=0))
    assert bound < 2 ** 53
    acc = qa.astype(np.float64) @ qw.astype(np.float64).T
    return acc.astype(np.int64)


def dequant(acc, s_a, s_w, bias=None):
    """Y_hat = s_a[i] * s_w[n] * acc[i, n] (+ b[n]), float64 (Eq. 3, z = 0)."""
    y = np.asarray(acc, dtype=np.float64) * np.asarray(s_a, dtype=np.float64)[:, None]
    y = y * np.asarray(s_w, dtype=np.float64)[None, :]
    if bias is not None:
        y = y + np.asarray(bias, dtype=np.float64)[None, :]
    return y


def sgat_linear_asym(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, qw, s_w, bias=None, bits=4):
    """Y_hat with asymmetric activation codes and symmetric weight codes:
    Y = s_a s_w sum_k (q_a - z_a) q_w (Eq. 3 and Eq. 5). Returns (Y float64
    [L, N], codes, s_a, z_a, acc int64 [L, N] = sum_k (q_a - z_a) q_w)."""
    codes, s_a, z_a = sgat_quantize_act_asym(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, bits)
    acc = int_gemm(codes - z_a[:, None], qw)
    return dequant(acc, s_a, s_w, bias), codes, s_a, z_a, acc


def sgat_linear(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, qw, s_w, bias=None, bits=4):
    """Y_hat of the state-guided quantised projection (Eq. 13), token order.

    For each state s: Y_hat^s = Q_a(Phi_s(X^s)) W_f, computed as the integer
    product of the codes followed by dequantisation; Y_hat^m and Y_hat^u are
    scattered back to their token positions. Returns (Y float64 [L, N],
    codes int32 [L, K], s_a float32 [L], acc int64 [L, N]).
    """
    X = np.asarray(X)
    L, K = X.shape
    N = np.asarray(qw).shape[0]
    g_m, g_u = state_gates(K, d_sh, d_m, d_u)
    I_m, I_u = state_index_sets(mask)
    Y = np.zeros((L, N), dtype=np.float64)
    codes = np.zeros((L, K), dtype=np.int32)
    s_a = np.zeros(L, dtype=F32)
    acc = np.zeros((L, N), dtype=np.int64)
    for I, a, g in ((I_m, a_m, g_m), (I_u, a_u, g_u)):
        if len(I) == 0:
            continue
        q, s = quantize_rows_sym(phi_state(X[I], a, g, hb), bits)
        acc_s = int_gemm(q, qw)
        Y[I] = dequant(acc_s, s, s_w, bias)
        codes[I] = q
        s_a[I] = s
        acc[I] = acc_s
    return Y, codes, s_a, acc
