"""Oracle: the quantised softmax-value product whose output TAC compensates
(Sec. 3.3: Z_hat, the quantised counterpart of Softmax(Q K^T / sqrt(d_h)) V,
corrected block-wise before the output projection), float64 unless stated.

Test infrastructure only (see the package docstring): the CUDA path never
imports this module.

The paper quantises the softmax-value multiplication but fixes neither its
bit widths nor its granularity. The readings here:

* scores per head h: s_ij = (q_i . k_j) / sqrt(d), with q, k the head's d
  channels of the query and key tokens;
* probabilities p_ij = e_ij / l_i, with e_ij = exp(s_ij - m_i),
  m_i = max_j s_ij and l_i = sum_j e_ij;
* P quantised per query row to unsigned 8 bits. The row's largest
  probability is 1 / l_i, so the scale is 1 / (255 l_i) and the code is
  c_ij = rne(p_ij * 255 l_i) = rne(255 e_ij);
* V quantised per channel (column c of the head) to signed 4 bits with the
  same symmetric quantiser as the activations (float32): t_c = amax_c / 7,
  v_jc = rne(V_jc * fl(7 / amax_c)). With a per-channel scale the sum over
  keys stays an integer sum;
* Z_hat_ic = (1 / (255 l_i)) * t_c * sum_j c_ij v_jc;
* TAC per head: Z_tac = Z_hat_h M_h^T + 1 d_h^T. The head's d channels are
  one TAC block (g = d).
* grouped-query attention (the Dream-7B / Qwen2.5 block): H query heads
  share Hkv key/value heads, query head h reading key/value head
  h // (H / Hkv); V is quantised per channel of the Hkv heads, so a group of
  query heads shares one set of V codes and scales.
"""

import numpy as np

from . import sgat, tac

F64 = np.float64


def scores(Qh, Kh, d):
    """s = Q_h K_h^T / sqrt(d) for one head (float64)."""
    return (np.asarray(Qh, F64) @ np.asarray(Kh, F64).T) / np.sqrt(d)


def p_codes(S):
    """Unsigned 8-bit per-row codes of softmax(S): c_ij = rne(255 exp(s_ij -
    m_i)) and the row sums l_i = sum_j exp(s_ij - m_i). Returns (codes int32
    [rows, keys], l float64 [rows])."""
    S = np.asarray(S, F64)
    m = S.max(axis=1, keepdims=True)
    e = np.exp(S - m)
    return np.rint(255.0 * e).astype(np.int32), e.sum(axis=1)


def v_codes(V):
    """Signed 4-bit per-channel codes of V [keys][channels]: the symmetric
    quantiser over each column. Returns (codes int32 [keys, channels],
    t float32 [channels])."""
    q, t = sgat.quantize_rows_sym(np.asarray(V, dtype=np.float32).T, 4)
    return q.T.copy(), t


def quantised_attention(Q, K, V, H, d, Hkv=None):
    """Z_hat [L][H d] for query tokens Q [L][H d] and key/value tokens K, V
    [L][Hkv d] (head h = channels h d .. h d + d - 1; query head h reads
    key/value head h // (H / Hkv); Hkv defaults to H).

    Returns (Z_hat float64, P codes int32 [H, L, L], l [H, L], V codes int32
    [L, Hkv d], t float32 [Hkv d], acc int64 [H, L, d]).
    """
    Q, K, V = (np.asarray(x) for x in (Q, K, V))
    Hkv = H if Hkv is None else Hkv
    assert H % Hkv == 0 and K.shape[1] == V.shape[1] == Hkv * d
    group = H // Hkv
    L = Q.shape[0]
    vq, t = v_codes(V)
    Z = np.empty((L, H * d), F64)
    codes = np.empty((H, L, L), np.int32)
    ls = np.empty((H, L), F64)
    acc = np.empty((H, L, d), np.int64)
    for h in range(H):
        ch = slice(h * d, (h + 1) * d)
        kv = slice((h // group) * d, (h // group + 1) * d)
        c, l = p_codes(scores(Q[:, ch], K[:, kv], d))
        a = sgat.int_gemm(c, vq[:, kv].T)
        codes[h], ls[h], acc[h] = c, l, a
        Z[:, ch] = a.astype(F64) / (255.0 * l[:, None]) * t[kv].astype(F64)[None, :]
    return Z, codes, ls, vq, t, acc


def attention_tac(Q, K, V, M, dvec, H, d, Hkv=None):
    """TAC of the quantised attention output: Z_hat M_h^T + 1 d_h^T per head
    (Eq. 17 with one block per head). Returns (Z_tac float64 [L][H d],
    Z_hat)."""
    Z = quantised_attention(Q, K, V, H, d, Hkv)[0]
    return tac.tac_apply(Z, M, dvec, d), Z
