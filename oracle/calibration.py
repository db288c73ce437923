"""Oracle: calibration of SGAT's dense orthogonal basis P (App. B, objective
Eq. 15 / the state-wise form of App. A), in float64 with torch's CPU
autograd.

Test infrastructure only (see the package docstring): the CUDA path never
imports this module. The GPU path runs on whatever basis this produces
(sgat_linear_dense takes P as an input).

App. B: P = [U_sh, U_m, U_u] starts as an orthogonalised Gaussian matrix and
stays orthogonal during calibration; only P is trained, layer by layer, on
paired full-precision and quantised outputs, with AdamW (learning rate 1e-3,
batch size 4, 15 epochs). The objective of one calibration sample (the
activations X_t of one denoising step, with its mask) is

    L = sum_s || X^s W^T - Q_a(X^s P G_s) Q_w(P^T W^T) ||_F^2      (Eq. 15)

Readings (the paper fixes none of these details):

* Orthogonality is kept by construction: P = P0 C(A), with P0 the
  orthogonalised Gaussian start (QR, columns signed so that R has a
  positive diagonal) and C(A) = (I - S)^-1 (I + S) the Cayley transform of
  the skew-symmetric S = A - A^T; A (d x d, zero at the start) is the
  trained parameter. Every P is orthogonal to round-off.
* The quantisers are the symmetric per-row (activations) and per-output-
  channel (weights) quantisers of Eq. 2 (scale amax / qmax); their rounding
  passes gradients straight through (the code's gradient is that of v / s),
  and the scale's gradient flows through the row maximum.
* "Batch size 4" is four calibration samples per AdamW step; an epoch is
  one pass over the samples in a seeded random order; AdamW's other
  settings are torch's defaults (betas 0.9 / 0.999, eps 1e-8, decoupled
  weight decay 0.01 on A); the mean of the four samples' L is minimised.
* The Hadamard smoothing of the other paths is not part of this basis: P
  here is the whole transform.
"""

import numpy as np

F64 = np.float64


def _torch():
    import torch
    return torch


def orthogonal_init(d, seed):
    """The orthogonalised Gaussian start: Q of the QR decomposition of a
    seeded N(0, 1) matrix, each column's sign chosen so that R's diagonal is
    positive (the unique orthogonal factor). float64 [d][d]."""
    G = np.random.default_rng(seed).standard_normal((d, d))
    Q, R = np.linalg.qr(G)
    return Q * np.sign(np.diag(R))[None, :]


def cayley(A):
    """C(A) = (I - S)^-1 (I + S) with S = A - A^T: orthogonal for every A
    (S skew-symmetric, so I - S is invertible). torch float64."""
    torch = _torch()
    S = A - A.T
    I = torch.eye(A.shape[0], dtype=A.dtype)
    return torch.linalg.solve(I - S, I + S)


def _quant_ste(v, bits):
    """Per-row symmetric quantisation v -> s * rne(v / s), s = amax / qmax,
    with the rounding passed straight through (torch, differentiable)."""
    torch = _torch()
    qmax = 2 ** (bits - 1) - 1
    amax = v.abs().amax(dim=1, keepdim=True)
    s = torch.where(amax > 0, amax / qmax, torch.ones_like(amax))
    u = v / s
    q = u + (torch.round(u) - u).detach()
    return torch.where(amax > 0, q * s, torch.zeros_like(v))


def gates(d, d_sh, d_m, d_u):
    """The 0/1 diagonals of G_m and G_u (Eq. 9), float64 [d] each."""
    assert d_sh + d_m + d_u == d
    g_m = np.concatenate([np.ones(d_sh), np.ones(d_m), np.zeros(d_u)])
    g_u = np.concatenate([np.ones(d_sh), np.zeros(d_m), np.ones(d_u)])
    return g_m, g_u


def state_objective(P, samples, W, d_sh, d_m, d_u, bits_a=4, bits_w=4):
    """Eq. 15 summed over the samples: for each sample (X [L][d], mask [L])
    and each state s with tokens, || X^s W^T - Q_a(X^s P G_s) Q_w(P^T W^T) ||_F^2.
    P, W: numpy or torch float64. Returns a torch scalar (differentiable in
    P when P is a torch tensor with gradients)."""
    torch = _torch()
    P = P if torch.is_tensor(P) else torch.as_tensor(np.asarray(P, F64))
    W = torch.as_tensor(np.asarray(W, F64))
    d = P.shape[0]
    g_m, g_u = (torch.as_tensor(g) for g in gates(d, d_sh, d_m, d_u))
    Wt = _quant_ste(W @ P, bits_w)                # rows of Q_w(P^T W^T)^T: per output channel
    total = torch.zeros((), dtype=torch.float64)
    for X, mask in samples:
        X = torch.as_tensor(np.asarray(X, F64))
        mask = np.asarray(mask)
        for state, g in ((1, g_m), (0, g_u)):
            idx = np.nonzero(mask == state)[0]
            if idx.size == 0:
                continue
            Xs = X[torch.as_tensor(idx)]
            Yfp = Xs @ W.T
            Yq = _quant_ste((Xs @ P) * g[None, :], bits_a) @ Wt.T
            total = total + ((Yfp - Yq) ** 2).sum()
    return total


def leakage(P, samples, d_sh, d_m, d_u):
    """sum over samples and states of || X^s P G_s^perp ||_F^2: the energy
    of each state's activations in the subspace its gate suppresses (the
    part of Delta_s = X^s P G_s^perp P^T W^T that does not depend on W,
    Eq. 28; zero exactly when Eq. 25's condition holds)."""
    P = np.asarray(P, F64)
    g_m, g_u = gates(P.shape[0], d_sh, d_m, d_u)
    tot = 0.0
    for X, mask in samples:
        X = np.asarray(X, F64)
        mask = np.asarray(mask)
        for state, g in ((1, g_m), (0, g_u)):
            Xs = X[mask == state]
            tot += float((((Xs @ P) * (1.0 - g)[None, :]) ** 2).sum())
    return tot


def calibrate_basis(samples, W, d_sh, d_m, d_u, bits_a=4, bits_w=4, lr=1e-3, batch=4, epochs=15,
                    weight_decay=0.01, seed=0, P0=None):
    """AdamW calibration of the orthogonal basis P on the Eq. 15 objective.

    samples: list of (X [L_t][d], mask [L_t]) calibration samples; W [N][d].
    Returns (P float64 [d][d], history) with history = dict(
      objective = full objective over all samples at the start and after
                  every epoch,
      orth_err  = max |P^T P - I| after every AdamW step,
      leakage   = leakage() at the start and after every epoch)."""
    torch = _torch()
    d = np.asarray(W).shape[1]
    P0 = orthogonal_init(d, seed) if P0 is None else np.asarray(P0, F64)
    P0t = torch.as_tensor(P0)
    A = torch.zeros((d, d), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([A], lr=lr, weight_decay=weight_decay)
    order_rng = np.random.default_rng(seed + 1)
    I = np.eye(d)

    def current():
        with torch.no_grad():
            return (P0t @ cayley(A)).numpy().copy()

    def full_objective(P):
        with torch.no_grad():
            return float(state_objective(torch.as_tensor(P), samples, W, d_sh, d_m, d_u, bits_a, bits_w))

    P = current()
    hist = dict(objective=[full_objective(P)], orth_err=[], leakage=[leakage(P, samples, d_sh, d_m, d_u)])
    for _ in range(epochs):
        order = order_rng.permutation(len(samples))
        for b0 in range(0, len(order), batch):
            chunk = [samples[i] for i in order[b0:b0 + batch]]
            opt.zero_grad()
            Pt = P0t @ cayley(A)
            loss = state_objective(Pt, chunk, W, d_sh, d_m, d_u, bits_a, bits_w) / len(chunk)
            loss.backward()
            opt.step()
            P = current()
            hist["orth_err"].append(float(np.abs(P.T @ P - I).max()))
        hist["objective"].append(full_objective(P))
        hist["leakage"].append(leakage(P, samples, d_sh, d_m, d_u))
    return P, hist
