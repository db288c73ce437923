"""Oracle: Temporal Attention Compensation (Sec. 3.3, App. C), float64.

Test infrastructure only (see the package docstring): the CUDA path never
imports this module.

``Z`` is the quantised attention representation Z_hat (N tokens x C
channels), split into B = C / g blocks of g channels. Block b's parameters
are ``M[b]`` (g x g, row r = output channel r of the block) and ``d[b]`` (g).
"""

import numpy as np

F64 = np.float64

# App. C default hyperparameters.
TAC_DEFAULTS = dict(g=16, rho=3e-4, eps=1e-8, eta=0.15, alpha=0.55,
                    eig_floor=1e-12, max_calib_samples=64)


def default_block_size(C, g_default=16):
    """Block size rule of App. C: g = 16, or if C is not divisible by 16, the
    largest block size not exceeding 16 that divides C."""
    for g in range(min(g_default, C), 0, -1):
        if C % g == 0:
            return g
    return 1


def tac_apply(Z, M, d, g):
    """Z_tac_b = Z_hat_b M_b^T + 1 d_b^T for b = 1..B (Eq. 17, App. C row-major
    form), in float64. Returns float64 [N, C]."""
    Z = np.asarray(Z, dtype=F64)
    N, C = Z.shape
    assert C % g == 0
    B = C // g
    M = np.asarray(M, dtype=F64).reshape(B, g, g)
    d = np.asarray(d, dtype=F64).reshape(B, g)
    out = np.empty((N, C), dtype=F64)
    for b in range(B):
        blk = slice(b * g, (b + 1) * g)
        out[:, blk] = Z[:, blk] @ M[b].T + d[b][None, :]
    return out


# ---------------------------------------------------------------------------
# Closed-form calibration (Eq. 18 and App. C)
# ---------------------------------------------------------------------------

def block_stats(Z, g):
    """Population mean and covariance of every g-block over the N flattened
    tokens (Eq. 30): mu_b = (1/N) sum_i z_ib, Sigma_b = (1/N) sum_i z_ib z_ib^T
    - mu_b mu_b^T. Returns (mu [B, g], Sigma [B, g, g])."""
    Z = np.asarray(Z, dtype=F64)
    N, C = Z.shape
    B = C // g
    Zb = Z.reshape(N, B, g)
    mu = Zb.mean(axis=0)
    second = np.einsum("nbi,nbj->bij", Zb, Zb) / N
    Sigma = second - np.einsum("bi,bj->bij", mu, mu)
    return mu, Sigma


def sym_power(A, p, floor=TAC_DEFAULTS["eig_floor"]):
    """A^p = Q diag(max(lambda_i, floor)^p) Q^T from the symmetric
    eigendecomposition A = Q diag(lambda) Q^T (App. C, matrix powers)."""
    A = np.asarray(A, dtype=F64)
    A = 0.5 * (A + A.T)
    lam, Q = np.linalg.eigh(A)
    lam = np.maximum(lam, floor) ** p
    return (Q * lam[None, :]) @ Q.T


def tac_calibrate(Z_fp, Z_q, g, rho=TAC_DEFAULTS["rho"], eps=TAC_DEFAULTS["eps"],
                  eta=TAC_DEFAULTS["eta"], alpha=TAC_DEFAULTS["alpha"]):
    """Closed-form TAC parameters from paired calibration activations.

    For each block: damping lambda_b = rho * max(Tr(Sigma^Q_b) / g, eps);
    M_b = (Sigma^FP_b)^(1/2) (Sigma^Q_b + lambda_b I)^(-1/2) (Eq. 18);
    singular values smoothed toward their mean, sigma' = (1 - eta) sigma +
    eta mean(sigma); shrinkage M_final = (1 - alpha) M_sv + alpha I; bias
    d_b = mu^FP_b - M_final mu^Q_b (App. C). Returns (M [B, g, g], d [B, g]).
    """
    mu_fp, S_fp = block_stats(Z_fp, g)
    mu_q, S_q = block_stats(Z_q, g)
    B = mu_fp.shape[0]
    I = np.eye(g)
    M_out = np.empty((B, g, g))
    d_out = np.empty((B, g))
    for b in range(B):
        lam = rho * max(np.trace(S_q[b]) / g, eps)
        M = sym_power(S_fp[b], 0.5) @ sym_power(S_q[b] + lam * I, -0.5)
        U, sig, Vt = np.linalg.svd(M)
        sig = (1.0 - eta) * sig + eta * sig.mean()
        M_sv = (U * sig[None, :]) @ Vt
        M_fin = (1.0 - alpha) * M_sv + alpha * I
        M_out[b] = M_fin
        d_out[b] = mu_fp[b] - M_fin @ mu_q[b]
    return M_out, d_out
