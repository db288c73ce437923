"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a
hand-worked fixture in tests/golden/, a closed form, brute force on tiny
inputs, or an identity of App. A. A plausible slip in the oracle (a dropped
term, a wrong sign, a swapped index or operand, a wrong rounding mode) fails
at least one of them.
"""

import itertools
import json
import math
import os

import numpy as np
import pytest

from oracle import sgat, tac
from tests.conftest import GOLDEN

F32 = np.float32
U32 = 2.0 ** -24


def golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ---------------------------------------------------------------------------
# Basis and fast transform (Eq. 8, Hadamard reading)
# ---------------------------------------------------------------------------

def test_hadamard_golden_h4():
    g = golden("hadamard_h4.json")
    H = sgat.hadamard_sylvester(4)
    assert H.tolist() == g["H4"]
    x = np.array(g["x"], dtype=F32)
    assert sgat.fwht_f32(x[None], 4)[0].tolist() == g["xH"]


@pytest.mark.parametrize("n", [1, 2, 8, 64, 512])
def test_hadamard_orthogonal_symmetric(n):
    H = sgat.hadamard_sylvester(n)
    assert np.array_equal(H, H.T)
    assert np.array_equal(H @ H.T, n * np.eye(n, dtype=np.int64))
    assert set(np.unique(H).tolist()) <= {-1, 1}


def brute_hadamard_entry(i, j):
    """Sylvester H_ij = (-1)^popcount(i & j), written independently."""
    return -1 if bin(i & j).count("1") % 2 else 1


@pytest.mark.parametrize("hb,K", [(2, 2), (8, 8), (16, 48), (256, 256), (512, 1536)])
def test_fwht_equals_dense_on_integers(hb, K):
    """On small integers every float32 butterfly is exact, so the fast
    transform must equal x @ blockdiag(H_hb) exactly."""
    rng = np.random.default_rng(hb + K)
    x = rng.integers(-8, 9, (5, K)).astype(F32)
    Hd = np.array([[brute_hadamard_entry(i, j) for j in range(hb)] for i in range(hb)], dtype=np.int64)
    BD = np.kron(np.eye(K // hb, dtype=np.int64), Hd)
    ref = x.astype(np.int64) @ BD
    out = sgat.fwht_f32(x, hb)
    assert np.array_equal(out.astype(np.int64), ref)


@pytest.mark.parametrize("hb", [64, 4096])
def test_fwht_float32_error_bound(hb):
    """Random normal input: each output is a sum of hb terms through log2(hb)
    float32 roundings, so |err| <= log2(hb) * u * sum|x| (u = 2^-24) plus
    second-order terms."""
    rng = np.random.default_rng(7)
    x = rng.standard_normal((3, hb)).astype(F32)
    ref = x.astype(np.float64) @ sgat.hadamard_sylvester(hb).astype(np.float64)
    out = sgat.fwht_f32(x, hb).astype(np.float64)
    bound = math.log2(hb) * U32 * np.abs(x).astype(np.float64).sum(axis=1, keepdims=True) * 1.01
    assert np.all(np.abs(out - ref) <= bound)


def test_fwht_involution():
    rng = np.random.default_rng(3)
    x = rng.integers(-100, 101, (4, 1024)).astype(F32)
    y = sgat.fwht_f32(sgat.fwht_f32(x, 1024), 1024)
    assert np.array_equal(y, 1024 * x)


# ---------------------------------------------------------------------------
# Gates (Eq. 9)
# ---------------------------------------------------------------------------

def test_gates_golden():
    g = golden("gates_k8.json")
    g_m, g_u = sgat.state_gates(g["K"], g["d_sh"], g["d_m"], g["d_u"])
    assert g_m.tolist() == g["g_m"]
    assert g_u.tolist() == g["g_u"]


def test_gates_partition():
    K, d_sh, d_m, d_u = 4096, 3840, 128, 128
    g_m, g_u = sgat.state_gates(K, d_sh, d_m, d_u)
    shared = g_m * g_u
    assert shared.sum() == d_sh and g_m.sum() == d_sh + d_m and g_u.sum() == d_sh + d_u
    assert np.all(g_m + g_u - shared == 1)   # the three subspaces cover d


# ---------------------------------------------------------------------------
# Quantiser (Eq. 2-3, symmetric reading)
# ---------------------------------------------------------------------------

def test_quant_golden():
    for c in golden("quant_examples.json")["cases"]:
        q, s = sgat.quantize_rows_sym(np.array([c["v"]], dtype=F32), c["bits"])
        assert q[0].tolist() == c["q"], c["name"]
        assert float(s[0]) == c["s"], c["name"]


def brute_quant_row(v, bits):
    """Independent restatement: pick q in [-qmax, qmax] nearest to the float32
    product p = fl32(v * r), ties to the even integer; distances exact in
    float64."""
    qmax = (1 << (bits - 1)) - 1
    amax = max(abs(float(t)) for t in v)
    if amax == 0:
        return [0] * len(v), 0.0
    r = np.float32(np.float32(qmax) / np.float32(amax))
    s = float(np.float32(np.float32(amax) / np.float32(qmax)))
    out = []
    for t in v:
        p = float(np.float32(np.float32(t) * r))
        best = None
        for q in range(-qmax, qmax + 1):
            dist = abs(p - q)
            key = (dist, q % 2)          # ties -> even
            if best is None or key < best[0]:
                best = (key, q)
        out.append(best[1])
    return out, s


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_quant_brute_force(bits):
    rng = np.random.default_rng(bits)
    for trial in range(300):
        n = int(rng.integers(1, 9))
        kind = trial % 3
        if kind == 0:
            v = rng.standard_normal(n)
        elif kind == 1:      # constructed near-ties: multiples of half a step
            v = rng.integers(-2 * ((1 << (bits - 1)) - 1), 2 * ((1 << (bits - 1)) - 1) + 1, n) * 0.5
        else:
            v = rng.standard_normal(n) * 10.0 ** rng.integers(-3, 4)
        v = v.astype(F32)
        q, s = sgat.quantize_rows_sym(v[None], bits)
        qb, sb = brute_quant_row(v, bits)
        assert q[0].tolist() == qb, (v, bits)
        assert float(s[0]) == sb


def test_quant_error_bound_and_extremes():
    rng = np.random.default_rng(11)
    v = (rng.standard_normal((64, 512)) * rng.lognormal(0, 2, (64, 1))).astype(F32)
    q, s = sgat.quantize_rows_sym(v, 4)
    assert np.all(np.abs(q) <= 7)
    err = np.abs(v.astype(np.float64) - q * s[:, None].astype(np.float64))
    assert np.all(err <= 0.5 * s[:, None] * (1 + 1e-5) + 1e-30)
    # the element of largest magnitude lands on +-qmax
    arg = np.argmax(np.abs(v), axis=1)
    assert np.all(np.abs(q[np.arange(64), arg]) == 7)


def test_pack_golden_and_roundtrip():
    g = golden("int4_packing.json")
    p = sgat.pack_int4(np.array([g["codes"]]))
    assert p[0].tolist() == g["bytes"]
    rng = np.random.default_rng(5)
    q = rng.integers(-8, 8, (7, 64))
    assert np.array_equal(sgat.unpack_int4(sgat.pack_int4(q)), q)


# ---------------------------------------------------------------------------
# Integer GEMM (Eq. 5 / Eq. 13)
# ---------------------------------------------------------------------------

def test_int_gemm_triple_loop():
    rng = np.random.default_rng(2)
    qa = rng.integers(-7, 8, (5, 96))
    qw = rng.integers(-7, 8, (6, 96))
    acc = sgat.int_gemm(qa, qw)
    for i, n in itertools.product(range(5), range(6)):
        s = 0
        for k in range(96):
            s += int(qa[i, k]) * int(qw[n, k])
        assert acc[i, n] == s


def test_int_gemm_extreme_accumulators():
    K = 18944
    qa = np.full((2, K), 7)
    qw = np.stack([np.full(K, 7), np.full(K, -7)])
    acc = sgat.int_gemm(qa, qw)
    assert acc[0, 0] == 49 * K and acc[0, 1] == -49 * K


# ---------------------------------------------------------------------------
# Quantised linear and the SGAT identities (Eq. 5, 6, 25-28)
# ---------------------------------------------------------------------------

def _case(L=24, K=256, N=40, seed=0):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((L, K)).astype(F32)
    X[:, 5] *= 12
    W = (rng.standard_normal((N, K)) * 0.05).astype(F32)
    mask = (rng.random(L) < 0.5).astype(np.uint8)
    return X, W, mask


def test_identity_transform_16bit_reproduces_fp_matmul():
    """P = I, all gates on, b = 16: Y_hat = Q_a(X) Q_w(W^T) must equal X W^T up
    to the quantisation error bound |x - x_hat| <= s_a/2, |w - w_hat| <= s_w/2
    (Eq. 5)."""
    X, W, mask = _case()
    K = X.shape[1]
    qw, s_w = sgat.prepare_weight(W, None, 1, 16)
    Y, codes, s_a, acc = sgat.sgat_linear(X, mask, None, None, 1, K, 0, 0, qw, s_w, bits=16)
    ref = X.astype(np.float64) @ W.astype(np.float64).T
    ea = 0.5 * s_a.astype(np.float64)[:, None]
    ew = 0.5 * s_w.astype(np.float64)[None, :]
    bound = (ea * np.abs(W).astype(np.float64).sum(1)[None, :]
             + ew * np.abs(X).astype(np.float64).sum(1)[:, None] + K * ea * ew)
    assert np.all(np.abs(Y - ref) <= bound * 1.0001 + 1e-12)
    assert np.linalg.norm(Y - ref) / np.linalg.norm(ref) < 2e-4


def test_transform_cancellation_full_precision():
    """Eq. 6 / Eq. 27 with G = I and a shared diagonal: (X P)(P^-1 W^T) = X W^T
    to float32 round-off, for both states."""
    X, W, mask = _case(K=512)
    K = X.shape[1]
    rng = np.random.default_rng(9)
    a = np.exp(rng.normal(0, 0.5, K)).astype(F32)
    V = sgat.sgat_transform(X, mask, a, a, 512, K, 0, 0).astype(np.float64)
    Wt = sgat.transform_weight_f32(W, (1.0 / a.astype(np.float64)).astype(F32), 512).astype(np.float64)
    Y = V @ Wt.T
    ref = X.astype(np.float64) @ W.astype(np.float64).T
    scale = np.abs(X).astype(np.float64) @ np.abs(W).astype(np.float64).T
    assert np.all(np.abs(Y - ref) <= 64 * 12 * U32 * scale + 1e-12)


def test_inactive_zero_condition_and_leakage():
    """App. A: if X^s P G_s^perp = 0 (Eq. 25) the gated transform reproduces
    X^s W^T; in general the difference equals Delta_s = X^s P G_s^perp P^T W^T
    (Eq. 28)."""
    L, K, N, hb = 16, 256, 24, 256
    rng = np.random.default_rng(4)
    d_m = d_u = K // 32
    d_sh = K - d_m - d_u
    g_m, g_u = sgat.state_gates(K, d_sh, d_m, d_u)
    a = np.exp(rng.normal(0, 0.3, K)).astype(F32)
    inv_a = (1.0 / a.astype(np.float64)).astype(F32)
    W = (rng.standard_normal((N, K)) * 0.05).astype(F32)
    H = sgat.hadamard_sylvester(hb).astype(np.float64)
    Wt = sgat.transform_weight_f32(W, inv_a, hb).astype(np.float64)
    for state, g in ((1, g_m), (0, g_u)):
        mask = np.full(L, state, np.uint8)
        # X^s built inside the active subspace: (X^s * a) H = U * g_s
        U = rng.standard_normal((L, K))
        Xs = (((U * g[None, :]) @ H / hb) / a.astype(np.float64)[None, :]).astype(F32)
        V = sgat.sgat_transform(Xs, mask, a, a, hb, d_sh, d_m, d_u).astype(np.float64)
        ref = Xs.astype(np.float64) @ W.astype(np.float64).T
        scale = np.abs(Xs).astype(np.float64) @ np.abs(W).astype(np.float64).T
        assert np.all(np.abs(V @ Wt.T - ref) <= 1e-5 * scale.max())
        # general X^s: the deviation is the leakage term of Eq. 28
        Xg = rng.standard_normal((L, K)).astype(F32)
        Vg = sgat.sgat_transform(Xg, mask, a, a, hb, d_sh, d_m, d_u).astype(np.float64)
        XP = (Xg.astype(np.float64) * a.astype(np.float64)) @ H
        delta = (XP * (1 - g[None, :])) @ (H / hb) @ (W.astype(np.float64) * inv_a.astype(np.float64)).T
        dev = Xg.astype(np.float64) @ W.astype(np.float64).T - Vg @ Wt.T
        scale = np.abs(Xg).astype(np.float64) @ np.abs(W).astype(np.float64).T
        assert np.all(np.abs(dev - delta) <= 1e-5 * scale.max())
        assert np.abs(delta).max() > 1e-3 * scale.max()   # the leakage is really there


def test_state_split_scatter():
    """Eq. 7 and the scatter after Eq. 13: each token is transformed with its
    own state's gate and smoothing, independent of the other tokens, and
    returns to its own position."""
    X, W, mask = _case(L=33, K=128, N=16, seed=3)
    K = X.shape[1]
    rng = np.random.default_rng(1)
    a_m = np.exp(rng.normal(0, 0.5, K)).astype(F32)
    a_u = np.exp(rng.normal(0, 0.5, K)).astype(F32)
    args = (a_m, a_u, 128, K - 8, 4, 4)
    codes, s_a = sgat.sgat_quantize_act(X, mask, *args, 4)
    # all-masked and all-unmasked runs give the per-state rows
    cm, sm = sgat.sgat_quantize_act(X, np.ones_like(mask), *args, 4)
    cu, su = sgat.sgat_quantize_act(X, np.zeros_like(mask), *args, 4)
    sel = mask[:, None] == 1
    assert np.array_equal(codes, np.where(sel, cm, cu))
    assert np.array_equal(s_a, np.where(mask == 1, sm, su))
    assert not np.array_equal(cm, cu)
    # permuting tokens permutes the result
    perm = rng.permutation(len(mask))
    cp, sp = sgat.sgat_quantize_act(X[perm], mask[perm], *args, 4)
    assert np.array_equal(cp, codes[perm]) and np.array_equal(sp, s_a[perm])


def test_weight_fold_scale_invariance():
    """Folding the exact 1/hb into the weight (Eq. 12) scales s_w by 1/hb and
    leaves every code unchanged."""
    _, W, _ = _case(N=32, K=512)
    q1, s1 = sgat.prepare_weight(W, None, 512, 4)
    q2, s2 = sgat.quantize_rows_sym(sgat.fwht_f32(W, 512), 4)
    assert np.array_equal(q1, q2)
    assert np.array_equal(s1, (s2 / F32(512)).astype(F32))


# ---------------------------------------------------------------------------
# TAC (Eq. 17, App. C)
# ---------------------------------------------------------------------------

def test_tac_golden():
    g = golden("tac_example.json")
    out = tac.tac_apply(np.array(g["z"]), np.array(g["M"]), np.array(g["d"]), g["g"])
    assert np.allclose(out, np.array(g["out"]), rtol=0, atol=1e-12)


def test_tac_identity_and_column_form():
    rng = np.random.default_rng(8)
    N, C, g = 5, 48, 16
    Z = rng.standard_normal((N, C))
    B = C // g
    eye = np.broadcast_to(np.eye(g), (B, g, g))
    assert np.array_equal(tac.tac_apply(Z, eye, np.zeros((B, g)), g), Z)
    M = rng.standard_normal((B, g, g))
    d = rng.standard_normal((B, g))
    out = tac.tac_apply(Z, M, d, g)
    # column-vector form z_b <- M_b z_b + d_b, written as explicit loops
    for i in range(N):
        for b in range(B):
            for r in range(g):
                s = d[b, r]
                for j in range(g):
                    s += M[b, r, j] * Z[i, b * g + j]
                assert abs(out[i, b * g + r] - s) <= 1e-12 * (1 + abs(s))


def test_tac_hyperparameters_and_block_rule():
    g = golden("hyperparameters.json")
    for k, v in g["tac"].items():
        assert tac.TAC_DEFAULTS[k] == v
    for C, expect in g["block_size_rule"]:
        assert tac.default_block_size(C) == expect


def test_tac_scalar_calibration_golden():
    g = golden("tac_scalar_calibration.json")
    M, d = tac.tac_calibrate(np.array(g["Z_fp"])[:, None], np.array(g["Z_q"])[:, None], 1,
                             rho=g["rho"], eps=g["eps"], eta=g["eta"], alpha=g["alpha"])
    assert abs(M[0, 0, 0] - g["M_final"]) < 1e-12
    assert abs(d[0, 0] - g["d"]) < 1e-12


def test_tac_calibration_invariants():
    rng = np.random.default_rng(12)
    N, C, g = 4096, 32, 16
    A = rng.standard_normal((C, C)) * 0.3 + np.eye(C)
    Z_fp = rng.standard_normal((N, C)) @ A.T + rng.normal(0, 1, C)
    Z_q = Z_fp * 0.9 + rng.standard_normal((N, C)) * 0.2 + 0.05
    # compensated mean equals the full-precision mean (bias estimation, App. C)
    M, d = tac.tac_calibrate(Z_fp, Z_q, g)
    out = tac.tac_apply(Z_q, M, d, g)
    assert np.allclose(out.mean(0), Z_fp.mean(0), atol=1e-10)
    # alpha = 1: the matrix degenerates to identity, only the mean is corrected
    M1, d1 = tac.tac_calibrate(Z_fp, Z_q, g, alpha=1.0)
    assert np.allclose(M1, np.eye(g)[None], atol=1e-12)
    assert np.allclose(d1.reshape(-1), Z_fp.mean(0) - Z_q.mean(0), atol=1e-12)
    # rho = eta = alpha = 0: covariance matching, M Sigma_Q M^T = Sigma_FP (Eq. 18)
    M0, _ = tac.tac_calibrate(Z_fp, Z_q, g, rho=0.0, eta=0.0, alpha=0.0)
    _, S_fp = tac.block_stats(Z_fp, g)
    _, S_q = tac.block_stats(Z_q, g)
    for b in range(C // g):
        assert np.allclose(M0[b] @ S_q[b] @ M0[b].T, S_fp[b], rtol=1e-8, atol=1e-9)
    # eta = 1: all singular values equal their mean before shrinkage
    Me, _ = tac.tac_calibrate(Z_fp, Z_q, g, eta=1.0, alpha=0.0)
    sv = np.linalg.svd(Me[0], compute_uv=False)
    assert np.allclose(sv, sv.mean(), rtol=1e-10)


def test_sym_power_closed_form():
    A = np.diag([4.0, 9.0, 0.0])
    R = np.array([[0.6, -0.8, 0], [0.8, 0.6, 0], [0, 0, 1.0]])
    B = R @ A @ R.T
    assert np.allclose(tac.sym_power(B, 0.5), R @ np.diag([2.0, 3.0, 1e-6]) @ R.T, atol=1e-12)
    assert np.allclose(tac.sym_power(B, -0.5), R @ np.diag([0.5, 1 / 3.0, 1e6]) @ R.T, rtol=1e-9)


def test_phi_state_dense_reference():
    """Phi_s(x) = ((x * a_s) H) G_s (Eq. 11) against a dense float64 product,
    with distinct smoothing per state and both states present."""
    L, K, hb = 20, 256, 128
    rng = np.random.default_rng(21)
    X = rng.standard_normal((L, K)).astype(F32)
    mask = (np.arange(L) % 3 == 0).astype(np.uint8)
    a_m = np.exp(rng.normal(0, 0.5, K)).astype(F32)
    a_u = np.exp(rng.normal(0, 0.5, K)).astype(F32)
    d_m = d_u = 8
    d_sh = K - 16
    g_m, g_u = sgat.state_gates(K, d_sh, d_m, d_u)
    BD = np.kron(np.eye(K // hb), sgat.hadamard_sylvester(hb).astype(np.float64))
    V = sgat.sgat_transform(X, mask, a_m, a_u, hb, d_sh, d_m, d_u).astype(np.float64)
    for i in range(L):
        a, g = (a_m, g_m) if mask[i] else (a_u, g_u)
        ref = ((X[i].astype(np.float64) * a.astype(np.float64)) @ BD) * g
        bound = 10 * U32 * (np.abs(X[i].astype(np.float64) * a) @ np.abs(BD)) + 1e-30
        assert np.all(np.abs(V[i] - ref) <= bound), i


def test_tac_singular_value_smoothing_formula():
    """App. C: M_sv keeps the singular vectors of M and maps every singular
    value to (1 - eta) sigma + eta mean(sigma)."""
    rng = np.random.default_rng(13)
    N, C, g = 2048, 16, 16
    A = rng.standard_normal((C, C)) * 0.5 + np.eye(C)
    Z_fp = rng.standard_normal((N, C)) @ A.T
    Z_q = Z_fp + rng.standard_normal((N, C)) * 0.3
    M0, _ = tac.tac_calibrate(Z_fp, Z_q, g, eta=0.0, alpha=0.0)
    for eta in (0.15, 1.0):
        Me, _ = tac.tac_calibrate(Z_fp, Z_q, g, eta=eta, alpha=0.0)
        s0 = np.linalg.svd(M0[0], compute_uv=False)
        se = np.linalg.svd(Me[0], compute_uv=False)
        assert np.allclose(se, (1 - eta) * s0 + eta * s0.mean(), rtol=1e-10)


# ---------------------------------------------------------------------------
# The quantised softmax-value product feeding TAC (oracle/attention.py)
# ---------------------------------------------------------------------------

def test_attention_p_codes_definition():
    """P's 8-bit codes: each row's largest probability 1 / l maps to 255;
    uniform scores give 255 everywhere and l = keys; every code is the
    nearest integer to 255 exp(s - m) by brute force over 0..255."""
    from oracle import attention as oatt
    c, l = oatt.p_codes(np.zeros((2, 7)))
    assert np.all(c == 255) and np.allclose(l, 7.0)
    rng = np.random.default_rng(3)
    S = rng.normal(0, 2, (5, 9))
    c, l = oatt.p_codes(S)
    assert np.all(c.max(axis=1) == 255)
    e = np.exp(S - S.max(axis=1, keepdims=True))
    assert np.allclose(l, e.sum(axis=1))
    brute = np.argmin(np.abs(255.0 * e[..., None] - np.arange(256)[None, None, :]), axis=-1)
    assert np.array_equal(c, brute)
    assert c.min() >= 0 and c.max() <= 255


def test_attention_v_codes_per_channel():
    """V's 4-bit codes run along each channel (column): every column with a
    non-zero entry reaches |code| 7, and codes are the brute-force nearest
    multiples of the column's step t = amax / 7."""
    from oracle import attention as oatt
    rng = np.random.default_rng(4)
    V = rng.normal(0, 1, (11, 6)).astype(np.float32)
    V[:, 2] *= 100.0                                   # one loud channel must not affect the others
    q, t = oatt.v_codes(V)
    assert q.shape == V.shape and t.shape == (6,)
    assert np.all(np.abs(q).max(axis=0) == 7)
    np.testing.assert_allclose(t, np.abs(V).max(axis=0) / 7, rtol=1e-6)
    brute = np.argmin(np.abs(V[..., None] / t[None, :, None] - np.arange(-7, 8)[None, None, :]), axis=-1) - 7
    assert np.array_equal(q, brute)


def test_attention_brute_force_tiny():
    """Z_hat against explicit loops over heads, queries, keys and channels
    (scores scaled by 1 / sqrt(d), codes per row / per channel)."""
    from oracle import attention as oatt
    rng = np.random.default_rng(5)
    L, H, d = 3, 2, 4
    Q, K, V = (rng.normal(0, 1, (L, H * d)).astype(np.float32) for _ in range(3))
    Z, codes, ls, vq, t, acc = oatt.quantised_attention(Q, K, V, H, d)
    for h in range(H):
        for i in range(L):
            s = [sum(float(Q[i, h * d + k]) * float(K[j, h * d + k]) for k in range(d)) / math.sqrt(d)
                 for j in range(L)]
            m = max(s)
            e = [math.exp(x - m) for x in s]
            lsum = sum(e)
            cs = [round(255.0 * x) for x in e]          # Python's round is half to even
            assert cs == list(codes[h, i]) and abs(lsum - ls[h, i]) < 1e-12
            for c in range(d):
                a = sum(cs[j] * int(vq[j, h * d + c]) for j in range(L))
                assert a == acc[h, i, c]
                want = a / (255.0 * lsum) * float(t[h * d + c])
                assert abs(want - Z[i, h * d + c]) <= 1e-12 * max(1.0, abs(want))


def test_attention_uniform_and_error_bound():
    """Q = 0 makes attention uniform: Z_hat is the mean of the dequantised
    V over keys exactly. For general inputs |Z_hat - softmax(s) V| stays
    within the rounding bound of 8-bit P and 4-bit V."""
    from oracle import attention as oatt
    rng = np.random.default_rng(6)
    L, H, d = 40, 2, 8
    K = rng.normal(0, 1, (L, H * d)).astype(np.float32)
    V = rng.normal(0, 1, (L, H * d)).astype(np.float32)
    Z, _, ls, vq, t, _ = oatt.quantised_attention(np.zeros_like(K), K, V, H, d)
    assert np.allclose(Z, (vq * t[None, :]).mean(axis=0)[None, :], rtol=1e-12, atol=1e-15)
    assert np.allclose(ls, L)
    Q = rng.normal(0, 1, (L, H * d)).astype(np.float32)
    Z, _, ls, _, t, _ = oatt.quantised_attention(Q, K, V, H, d)
    for h in range(H):
        ch = slice(h * d, (h + 1) * d)
        S = oatt.scores(Q[:, ch], K[:, ch], d)
        P = np.exp(S - S.max(axis=1, keepdims=True))
        P /= P.sum(axis=1, keepdims=True)
        exact = P @ V[:, ch].astype(np.float64)
        vmax = np.abs(V[:, ch]).max(axis=0)
        bound = (t[ch][None, :] / 2) * (1 + L / (510 * ls[h][:, None])) + L * vmax[None, :] / (510 * ls[h][:, None])
        assert np.all(np.abs(Z[:, ch] - exact) <= bound + 1e-12)


def test_attention_gqa_equals_mha_on_repeated_heads():
    """Grouped-query attention with H query heads over Hkv key/value heads
    equals multi-head attention whose K and V repeat every key/value head
    H / Hkv times (query head h reads key/value head h // (H / Hkv)): the
    repeated channels carry identical columns, so their per-channel V codes
    and scales are identical too. Swapping the group order (a plausible
    indexing slip, h % Hkv) gives a different result."""
    from oracle import attention as oatt
    rng = np.random.default_rng(17)
    L, H, Hkv, d = 24, 6, 2, 8
    Q = rng.normal(0, 1, (L, H * d)).astype(np.float32)
    K, V = (rng.normal(0, 1, (L, Hkv * d)).astype(np.float32) for _ in range(2))
    rep = np.concatenate([np.arange(k * d, (k + 1) * d) for k in np.repeat(np.arange(Hkv), H // Hkv)])
    Zg, cg, lg, vqg, tg, ag = oatt.quantised_attention(Q, K, V, H, d, Hkv)
    Zm, cm, lm, vqm, tm, am = oatt.quantised_attention(Q, K[:, rep], V[:, rep], H, d)
    assert np.array_equal(cg, cm) and np.array_equal(ag, am) and np.array_equal(lg, lm)
    assert np.array_equal(Zg, Zm) and np.array_equal(tg[rep], tm) and np.array_equal(vqg[:, rep], vqm)
    wrong = np.concatenate([np.arange(k * d, (k + 1) * d) for k in np.tile(np.arange(Hkv), H // Hkv)])
    Zw = oatt.quantised_attention(Q, K[:, wrong], V[:, wrong], H, d)[0]
    assert not np.allclose(Zg, Zw)


def test_attention_tac_identity():
    """TAC with M = I and d = 0 returns Z_hat unchanged (P6 on this path)."""
    from oracle import attention as oatt
    rng = np.random.default_rng(7)
    L, H, d = 16, 2, 8
    Q, K, V = (rng.normal(0, 1, (L, H * d)).astype(np.float32) for _ in range(3))
    M = np.broadcast_to(np.eye(d), (H, d, d))
    Zt, Z = oatt.attention_tac(Q, K, V, M, np.zeros((H, d)), H, d)
    assert np.array_equal(Zt, Z)


# ---------------------------------------------------------------------------
# Asymmetric activation quantiser (Eq. 2-4) and its linear
# ---------------------------------------------------------------------------

def test_asym_quant_worked_example():
    """Eq. 4 on v = (-1, 0.5, 2, 0), b = 4, worked by hand: X_max - X_min = 3,
    s = 3/15 = 0.2, X / s = 5 v, z = round(1 / 0.2) = 5; Eq. 2 gives
    round(-5) + 5 = 0, round(2.5) + 5 = 2 + 5 (half to even), round(10) + 5 =
    15, 0 + 5 = 5."""
    q, s, z = sgat.quantize_rows_asym(np.array([[-1.0, 0.5, 2.0, 0.0]], F32), 4)
    assert q.tolist() == [[0, 7, 15, 5]] and z.tolist() == [5]
    assert s[0] == F32(0.2)


def _brute_asym_row(a, k, m, bits):
    """Row with X_min = -a 2^-k, X_max = (L - a) 2^-k (L = 2^b - 1) and inner
    values m 2^-k / 2, all exact: v / s = v 2^k is exact. The code of v is the
    integer of [0, L] minimising |s (q - z) - v| = 2^-k |q - a - v 2^k|,
    ties to the even integer before the shift by z = a, which is Eq. 2 with
    round-half-even."""
    levels = (1 << bits) - 1
    vals = [-a, levels - a] + [mm / 2 for mm in m]
    v = np.array([x * 2.0 ** -k for x in vals], dtype=F32)
    want = []
    for x in vals:
        best = None
        for n in range(-2 * levels, 2 * levels + 1):            # n = round(v / s) candidate
            d = abs(n - x)
            if best is None or d < best[0] - 1e-12 or (abs(d - best[0]) <= 1e-12 and n % 2 == 0):
                best = (d, n)
        want.append(min(max(best[1] + a, 0), levels))
    return v, want, a


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_asym_quant_brute_force(bits):
    rng = np.random.default_rng(40 + bits)
    levels = (1 << bits) - 1
    for _ in range(60):
        a = int(rng.integers(0, levels + 1))
        k = int(rng.integers(-3, 6))
        m = rng.integers(-2 * a, 2 * (levels - a) + 1, 9)
        v, want, z_want = _brute_asym_row(a, k, m, bits)
        q, s, z = sgat.quantize_rows_asym(v[None], bits)
        assert q[0].tolist() == want and z[0] == z_want, (a, k, m.tolist(), bits)
        assert s[0] == F32(2.0 ** -k)


def test_asym_quant_invariants():
    """Random rows: codes in [0, 15], z in [0, 15]; dequantisation (Eq. 3)
    within half a step (no clamping: the range holds every value); an
    all-zero row gives s = 0, z = 0, codes 0; a row with X_max = -X_min has
    z = round(7.5) = 8; a row of positive values has z = 0 (zero is in the
    range)."""
    rng = np.random.default_rng(7)
    v = (rng.standard_normal((64, 96)) * rng.uniform(0.01, 10, (64, 1))).astype(F32)
    v[3] = 0
    v[5] = np.abs(v[5])
    v[6, :2] = [2.5, -2.5]
    v[6, 2:] = np.clip(v[6, 2:], -2.5, 2.5)
    q, s, z = sgat.quantize_rows_asym(v, 4)
    assert q.min() >= 0 and q.max() <= 15 and z.min() >= 0 and z.max() <= 15
    deq = s.astype(np.float64)[:, None] * (q - z[:, None])
    assert np.all(np.abs(deq - v) <= 0.5 * s.astype(np.float64)[:, None] * (1 + 1e-5) + 1e-30)
    assert s[3] == 0 and z[3] == 0 and not q[3].any()
    assert z[5] == 0 and q[5].min() == 0
    assert z[6] == 8


def test_asym_linear_16bit_reproduces_fp_matmul():
    """P = I, all gates on, b = 16 for both quantisers: Y_hat = s_a s_w
    sum_k (q_a - z_a) q_w must equal X W^T within the quantisation bound.
    Dropping the zero point, or subtracting it with the wrong sign, misses
    by the size of z times the weight row sums."""
    X, W, mask = _case()
    K = X.shape[1]
    qw, s_w = sgat.prepare_weight(W, None, 1, 16)
    Y, codes, s_a, z_a, acc = sgat.sgat_linear_asym(X, mask, None, None, 1, K, 0, 0, qw, s_w, bits=16)
    ref = X.astype(np.float64) @ W.astype(np.float64).T
    ea = 0.5 * s_a.astype(np.float64)[:, None]
    ew = 0.5 * s_w.astype(np.float64)[None, :]
    bound = (ea * np.abs(W).astype(np.float64).sum(1)[None, :]
             + ew * np.abs(X).astype(np.float64).sum(1)[:, None] + K * ea * ew)
    assert np.all(np.abs(Y - ref) <= bound * 1.0001 + 1e-12)
    assert np.linalg.norm(Y - ref) / np.linalg.norm(ref) < 2e-4
    assert z_a.max() > 1000                                  # the zero point matters here


def test_asym_linear_triple_loop():
    """acc = sum_k (q_a - z_a) q_w by explicit loops on a tiny case."""
    rng = np.random.default_rng(3)
    X = rng.standard_normal((5, 16)).astype(F32)
    W = rng.standard_normal((3, 16)).astype(F32)
    qw, s_w = sgat.prepare_weight(W, None, 16, 4)
    mask = np.array([0, 1, 0, 1, 1], np.uint8)
    Y, codes, s_a, z_a, acc = sgat.sgat_linear_asym(X, mask, None, None, 16, 8, 4, 4, qw, s_w)
    for i in range(5):
        for n in range(3):
            want = sum((int(codes[i, k]) - int(z_a[i])) * int(qw[n, k]) for k in range(16))
            assert acc[i, n] == want
            assert Y[i, n] == float(want) * float(s_a[i]) * float(s_w[n])


# ---------------------------------------------------------------------------
# Dense basis (the learned orthogonal P of App. B) as a 16-bit product
# ---------------------------------------------------------------------------

def test_dense_basis_permutation_is_exact():
    """A permutation is orthogonal and exact in float16: the dense path then
    permutes the float16-rounded scaled rows and quantises them, which a
    direct computation gives exactly."""
    rng = np.random.default_rng(8)
    L, K = 12, 64
    X = rng.standard_normal((L, K)).astype(F32)
    perm = rng.permutation(K)
    P = np.zeros((K, K), np.float16)
    P[perm, np.arange(K)] = 1                        # (x P)[j] = x[perm[j]]
    mask = np.zeros(L, np.uint8)
    codes, s, V = sgat.sgat_quantize_act_dense(X, mask, None, None, P, K, 0, 0)
    want = X.astype(np.float16).astype(F32)[:, perm]
    assert np.array_equal(V, want)
    q, s2 = sgat.quantize_rows_sym(want, 4)
    assert np.array_equal(codes, q) and np.array_equal(s, s2)


def test_dense_basis_matches_fast_hadamard_on_exact_inputs():
    """P = H_4 / 2 (block-diagonal, orthogonal, entries +-1/2 exact in
    float16) on small-integer inputs: every value is exact in both paths, so
    the dense product equals the fast transform of hb = 4 scaled by 1/2."""
    rng = np.random.default_rng(9)
    L, K = 6, 32
    X = rng.integers(-8, 9, (L, K)).astype(F32)
    H4 = sgat.hadamard_sylvester(4).astype(np.float64)
    P = np.kron(np.eye(K // 4), H4 / 2).astype(np.float16)
    V = sgat.dense_basis_product(X, P)
    assert np.array_equal(V, sgat.fwht_f32(X, 4) * F32(0.5))


def test_dense_basis_cancellation_16bit():
    """A random orthogonal P (QR of a Gaussian, rounded to float16): the
    16-bit dense linear reproduces X W^T up to the float16 roundings of the
    transform. Applying P^T instead of P on one side, or P on both sides
    transposed, breaks the cancellation by order one."""
    rng = np.random.default_rng(10)
    L, K, N = 16, 128, 24
    X = rng.standard_normal((L, K)).astype(F32)
    W = (rng.standard_normal((N, K)) * 0.1).astype(F32)
    Q, _ = np.linalg.qr(rng.standard_normal((K, K)))
    P = Q.astype(np.float16)
    mask = (rng.random(L) < 0.5).astype(np.uint8)
    codes, s_a, _ = sgat.sgat_quantize_act_dense(X, mask, None, None, P, K, 0, 0, bits=16)
    qw, s_w, _ = sgat.prepare_weight_dense(W, None, P, bits=16)
    Y = sgat.dequant(sgat.int_gemm(codes, qw), s_a, s_w)
    ref = X.astype(np.float64) @ W.astype(np.float64).T
    assert np.linalg.norm(Y - ref) / np.linalg.norm(ref) < 4e-3
    qt, st, _ = sgat.prepare_weight_dense(W, None, P.T.copy(), bits=16)
    Yt = sgat.dequant(sgat.int_gemm(codes, qt), s_a, st)
    assert np.linalg.norm(Yt - ref) / np.linalg.norm(ref) > 0.5


# ---------------------------------------------------------------------------
# Block glue (RMSNorm, rotary embedding, SwiGLU): standard definitions
# ---------------------------------------------------------------------------

def test_rmsnorm_worked_example_and_invariants():
    """h = (3, 4): mean square 12.5, so y = h / sqrt(12.5) * w (by hand:
    (0.848528..., 1.131370...) for w = 1). A constant row c gives w * c /
    |c| up to eps; scaling a row does not change its normalised values
    (eps = 0); the gain multiplies per column (a transposed gain fails)."""
    from oracle import glue
    y = glue.rmsnorm([[3.0, 4.0]], [1.0, 1.0], 0.0)
    assert np.allclose(y, [[3 / math.sqrt(12.5), 4 / math.sqrt(12.5)]], rtol=1e-15)
    assert abs(y[0, 0] - 0.8485281374238570) < 1e-15 and abs(y[0, 1] - 1.1313708498984760) < 1e-15
    w = np.array([0.5, 2.0, -1.0, 3.0])
    assert np.allclose(glue.rmsnorm(np.full((1, 4), -2.5), w, 1e-12), -w[None, :], atol=1e-12)
    rng = np.random.default_rng(3)
    h = rng.normal(0, 1, (5, 16))
    w = rng.normal(1, 0.1, 16)
    assert np.allclose(glue.rmsnorm(7.0 * h, w, 0.0), glue.rmsnorm(h, w, 0.0), rtol=1e-13)
    y = glue.rmsnorm(h, w, 0.0)
    assert np.allclose(np.mean((y / w[None, :]) ** 2, axis=1), 1.0, rtol=1e-13)


def test_rope_identity_rotation_and_composition():
    """Position 0 is the identity; each rotated pair keeps its norm; two
    rotations compose (rotating by p1 then p2 equals rotating by p1 + p2);
    the first frequency is 1, so pair 0 turns by pos radians (worked by hand
    at pos = 1: (1, 0) -> (cos 1, sin 1)); columns past the rotated heads
    are untouched."""
    from oracle import glue
    rng = np.random.default_rng(4)
    L, heads, d = 6, 3, 128
    x = rng.normal(0, 1, (L, heads * d + 64))
    assert np.array_equal(glue.rope(x, np.zeros(L), heads, 1e6), x)
    pos = rng.integers(0, 2048, L)
    y = glue.rope(x, pos, heads, 1e6)
    for h in range(heads):
        a, b = x[:, h * d:h * d + 64], x[:, h * d + 64:(h + 1) * d]
        ya, yb = y[:, h * d:h * d + 64], y[:, h * d + 64:(h + 1) * d]
        assert np.allclose(a * a + b * b, ya * ya + yb * yb, rtol=1e-12)
    p1, p2 = rng.integers(0, 1000, L), rng.integers(0, 1000, L)
    assert np.allclose(glue.rope(glue.rope(x, p1, heads, 1e4), p2, heads, 1e4),
                       glue.rope(x, p1 + p2, heads, 1e4), atol=1e-9)
    assert np.array_equal(y[:, heads * d:], x[:, heads * d:])
    e = np.zeros((1, d))
    e[0, 0] = 1.0
    r = glue.rope(e, [1], 1, 1e6)
    assert abs(r[0, 0] - math.cos(1.0)) < 1e-15 and abs(r[0, 64] - math.sin(1.0)) < 1e-15
    assert glue.rope_frequencies(1e6)[0] == 1.0
    assert abs(glue.rope_frequencies(1e6)[32] - 1e6 ** -0.5) < 1e-18


def test_swiglu_values():
    """silu(0) = 0, silu(x) -> x for large x, silu(-x) = silu(x) - x."""
    from oracle import glue
    x = np.array([0.0, 30.0, -2.0, 1.5])
    s = glue.swiglu(x, np.ones(4))
    assert s[0] == 0.0 and abs(s[1] - 30.0) < 1e-11
    assert abs(glue.swiglu([2.0], [1.0])[0] - glue.swiglu([-2.0], [1.0])[0] - 2.0) < 1e-15
    assert abs(s[3] - 1.5 / (1 + math.exp(-1.5))) < 1e-15


# ---------------------------------------------------------------------------
# Calibration of the dense orthogonal basis (App. B, Eq. 15)
# ---------------------------------------------------------------------------

def test_cayley_map_is_orthogonal():
    """C(0) = I; C(A) is orthogonal with determinant +1 for any A; a
    transposed solve (C = (I + S)(I - S)^-1 computed wrongly as (I + S)^-1
    (I - S)) would give C(A)^T instead, so C(A) is checked against the
    explicit formula on a worked 2 x 2 case: S = [[0, -t], [t, 0]] gives the
    rotation by 2 atan(t)."""
    import torch
    from oracle import calibration as oc
    assert torch.equal(oc.cayley(torch.zeros(5, 5, dtype=torch.float64)), torch.eye(5, dtype=torch.float64))
    A = torch.as_tensor(np.random.default_rng(2).normal(0, 1, (7, 7)))
    C = oc.cayley(A).numpy()
    assert np.abs(C.T @ C - np.eye(7)).max() < 1e-13 and abs(np.linalg.det(C) - 1.0) < 1e-12
    t = 0.3
    C2 = oc.cayley(torch.tensor([[0.0, 0.0], [t, 0.0]], dtype=torch.float64)).numpy()   # S = [[0, -t], [t, 0]]
    th = 2 * math.atan(t)
    assert np.allclose(C2, [[math.cos(th), -math.sin(th)], [math.sin(th), math.cos(th)]], atol=1e-15)


def test_state_objective_brute_force():
    """Eq. 15 against explicit numpy loops on a tiny case: per state, the
    gated transformed rows quantised per row, the weight quantised per
    output channel of P^T W^T, the squared Frobenius error summed."""
    from oracle import calibration as oc
    rng = np.random.default_rng(8)
    d, N = 8, 5
    d_sh, d_m, d_u = 4, 2, 2
    P = oc.orthogonal_init(d, 3)
    W = rng.normal(0, 1, (N, d))
    samples = [(rng.normal(0, 1, (6, d)), np.array([1, 0, 1, 1, 0, 0])), (rng.normal(0, 1, (3, d)), np.array([0, 0, 0]))]
    g_m, g_u = oc.gates(d, d_sh, d_m, d_u)

    def q_rows(v, bits):
        qmax = 2 ** (bits - 1) - 1
        out = np.zeros_like(v)
        for i in range(v.shape[0]):
            a = np.abs(v[i]).max()
            if a > 0:
                s = a / qmax
                out[i] = np.array([round(x / s) for x in v[i]]) * s      # half to even
        return out
    Wt = q_rows(W @ P, 4)
    want = 0.0
    for X, mask in samples:
        for state, g in ((1, g_m), (0, g_u)):
            Xs = X[mask == state]
            if len(Xs):
                want += float(((Xs @ W.T - q_rows((Xs @ P) * g[None, :], 4) @ Wt.T) ** 2).sum())
    got = float(oc.state_objective(P, samples, W, d_sh, d_m, d_u))
    assert abs(got - want) <= 1e-10 * want


def test_calibration_recovers_planted_subspaces():
    """Activations built to satisfy Eq. 25 for a planted basis P*: masked
    tokens live in span(U*_sh, U*_m), unmasked ones in span(U*_sh, U*_u).
    With 16-bit quantisers and an orthogonal W the objective is the energy
    of Delta_s of Eq. 28, || X^s P G_s^perp P^T W^T ||^2 = || X^s P G_s^perp ||^2
    (the leakage), up to rounding; so calibration from a random orthogonal
    start must drive the leakage toward zero: below 2% of its start, with P
    orthogonal to round-off after every step and the objective below its
    start after every epoch. (With a general W the objective can also fall
    by hiding the leakage in W's small singular directions.)"""
    from oracle import calibration as oc
    rng = np.random.default_rng(11)
    d, d_sh, d_m, d_u = 16, 12, 2, 2
    Ps = oc.orthogonal_init(d, 99)
    Um, Uu, Ush = Ps[:, d_sh:d_sh + d_m], Ps[:, d_sh + d_m:], Ps[:, :d_sh]
    samples = []
    for _ in range(8):
        mask = (rng.random(24) < 0.5).astype(np.uint8)
        X = np.empty((24, d))
        for i in range(24):
            B = np.concatenate([Ush, Um if mask[i] else Uu], axis=1)
            X[i] = B @ rng.normal(0, 1, d_sh + d_m)
        samples.append((X, mask))
    W = 2.0 * oc.orthogonal_init(d, 7)
    P, hist = oc.calibrate_basis(samples, W, d_sh, d_m, d_u, bits_a=16, bits_w=16, lr=2e-2, epochs=80, seed=5)
    assert max(hist["orth_err"]) < 1e-12
    assert oc.leakage(Ps, samples, d_sh, d_m, d_u) < 1e-20            # the planted basis has none
    assert hist["leakage"][-1] < 0.02 * hist["leakage"][0]
    assert all(o <= hist["objective"][0] for o in hist["objective"][1:])


def test_calibration_paper_settings_reduce_objective():
    """App. B's settings (AdamW lr 1e-3, batch 4, 15 epochs, 4-bit codes) on
    the synthetic calibration set: P stays orthogonal to round-off after
    every step, starts at the orthogonalised Gaussian (the objective's first
    entry is the objective of that start), and the objective after every
    epoch is below its value at the start."""
    from oracle import calibration as oc
    from paper_2606_04945_gb300 import inputs
    d = 64
    samples, W = inputs.basis_calibration_set(4, d, n_samples=8, tokens=32)
    d_m = d_u = d // 32
    d_sh = d - 2 * d_m
    P, hist = oc.calibrate_basis(samples, W, d_sh, d_m, d_u, seed=1)
    assert len(hist["orth_err"]) == 15 * 2 and max(hist["orth_err"]) < 1e-12
    start = float(oc.state_objective(oc.orthogonal_init(d, 1), samples, W, d_sh, d_m, d_u))
    assert abs(hist["objective"][0] - start) <= 1e-12 * start
    assert all(o < hist["objective"][0] for o in hist["objective"][1:])
