"""tac_calibrate on the GPU against the oracle's closed-form calibration
(App. C) and against the invariants that fix it (the P7 pins).

Paired calibration activations are synthetic. Z_fp has correlated channels
inside each block and per-channel means (a random g x g mixing of Gaussian
tokens). Z_q is Z_fp quantised per token to 4 bits and dequantised, plus
small noise: the kind of error TAC compensates. Both are stored in the
test's 16- or 32-bit type, and the oracle reads the same values in
float64.

Tolerance: the kernel works in float64 with the eigenvectors accumulated
in float32, and writes float32. So M is compared to 2e-5 of its largest
entry, and d to 2e-5 of the scale of mu^FP and M mu^Q.
"""

import numpy as np
import pytest
import torch

from oracle import tac as otac
from tests import helpers as H


def paired(seed, N, C, g, dtype):
    rng = np.random.default_rng(seed)
    B = C // g
    X = rng.standard_normal((N, B, g))
    mix = rng.standard_normal((B, g, g)) / np.sqrt(g) + np.eye(g)[None]
    Z = np.einsum("nbi,bij->nbj", X, mix).reshape(N, C) + rng.normal(0, 0.5, C)[None, :]
    amax = np.abs(Z).max(axis=1, keepdims=True)
    s = amax / 7.0
    Zq = np.clip(np.rint(Z / s), -7, 7) * s + rng.normal(0, 0.01, Z.shape)
    cast = {"f16": np.float16, "bf16": None, "f32": np.float32}[dtype]
    if dtype == "bf16":
        from paper_2606_04945_gb300 import inputs
        return inputs.round_to_bf16(Z.astype(np.float32)), inputs.round_to_bf16(Zq.astype(np.float32))
    return Z.astype(cast).astype(np.float32), Zq.astype(cast).astype(np.float32)


def run_gpu(abi, Zf, Zq, g, dtype, **hp):
    N, C = Zf.shape
    dt = H.torch_dtype(dtype)
    M = torch.empty(C // g, g, g, dtype=torch.float32, device="cuda")
    d = torch.empty(C // g, g, dtype=torch.float32, device="cuda")
    abi.tac_calibrate(H.dev(Zf, dt), H.dev(Zq, dt), g, M, d, **hp)
    abi.check_status()
    return M.cpu().numpy().astype(np.float64), d.cpu().numpy().astype(np.float64)


def close(Mg, dg, Mo, do, Zf, Zq, g):
    mu_fp, _ = otac.block_stats(Zf, g)
    mu_q, _ = otac.block_stats(Zq, g)
    scale_M = max(1.0, np.abs(Mo).max())
    err_M = np.abs(Mg - Mo).max() / scale_M
    scale_d = np.abs(mu_fp).max() + np.abs(np.einsum("bij,bj->bi", Mo, mu_q)).max() + 1e-30
    err_d = np.abs(dg - do).max() / scale_d
    return err_M, err_d


@pytest.mark.gpu
@pytest.mark.parametrize("N,C,g,dtype,hp", [
    (1000, 256, 16, "f16", {}),                                    # the paper's default block size
    (1024, 4096, 128, "f16", {}),                                  # the LLaDA attention width, g = 128
    (300, 512, 64, "bf16", dict(rho=1e-3, eta=0.3, alpha=0.2)),
    (77, 128, 4, "f32", {}),
    (8, 64, 16, "f16", {}),                                        # fewer tokens than channels: singular Sigma
])
def test_tac_calibrate_matches_oracle(abi, N, C, g, dtype, hp):
    Zf, Zq = paired(N + C + g, N, C, g, dtype)
    Mg, dg = run_gpu(abi, Zf, Zq, g, dtype, **hp)
    Mo, do = otac.tac_calibrate(Zf, Zq, g, **hp)
    err_M, err_d = close(Mg, dg, Mo, do, Zf, Zq, g)
    assert err_M <= 2e-5, f"M differs by {err_M:.3g} of its scale"
    assert err_d <= 2e-5, f"d differs by {err_d:.3g} of its scale"


@pytest.mark.gpu
def test_tac_calibrate_invariants(abi):
    """P7 on the GPU's parameters:
    - alpha = 1 leaves only the mean correction (M = I, d = mu_fp - mu_q);
    - the compensated quantised tokens have the full-precision mean;
    - with rho = eta = alpha = 0, M Sigma^Q M^T = Sigma^FP."""
    N, C, g = 512, 256, 32
    Zf, Zq = paired(5, N, C, g, "f32")
    mu_fp, S_fp = otac.block_stats(Zf, g)
    mu_q, S_q = otac.block_stats(Zq, g)
    M1, d1 = run_gpu(abi, Zf, Zq, g, "f32", alpha=1.0)
    assert np.array_equal(M1, np.broadcast_to(np.eye(g), M1.shape))
    assert np.abs(d1 - (mu_fp - mu_q)).max() <= 1e-6 * (1 + np.abs(mu_fp).max())
    M, d = run_gpu(abi, Zf, Zq, g, "f32")
    out = otac.tac_apply(Zq, M, d, g)
    assert np.abs(out.mean(axis=0).reshape(-1, g) - mu_fp).max() <= 1e-5 * (1 + np.abs(mu_fp).max())
    M0, _ = run_gpu(abi, Zf, Zq, g, "f32", rho=0.0, eta=0.0, alpha=0.0)
    lhs = np.einsum("bij,bjk,blk->bil", M0, S_q, M0)
    assert np.abs(lhs - S_fp).max() <= 1e-4 * np.abs(S_fp).max()


@pytest.mark.gpu
def test_tac_calibrate_drives_tac_apply(abi):
    """The calibrated parameters feed tac_apply directly (same layout): the
    GPU's TAC of Z_q with its own calibration matches the oracle's TAC with
    the oracle's calibration, and moves Z_q's block statistics toward
    Z_fp's."""
    N, C, g = 1024, 512, 128
    Zf, Zq = paired(9, N, C, g, "f16")
    Mg, dg = run_gpu(abi, Zf, Zq, g, "f16")
    Mt = torch.from_numpy(Mg.astype(np.float32)).cuda()
    dt_ = torch.from_numpy(dg.astype(np.float32)).cuda()
    out = torch.empty(N, C, dtype=torch.float32, device="cuda")
    abi.tac_apply(H.dev(Zq, torch.float16), Mt, dt_, g, out)
    abi.check_status()
    Mo, do = otac.tac_calibrate(Zf, Zq, g)
    ref = otac.tac_apply(Zq, Mo, do, g)
    got = out.cpu().numpy().astype(np.float64)
    assert np.abs(got - ref).max() <= 1e-4 * np.abs(ref).max()
    _, S_fp = otac.block_stats(Zf, g)
    _, S_q = otac.block_stats(Zq, g)
    _, S_t = otac.block_stats(got, g)
    assert np.linalg.norm(S_t - S_fp) < np.linalg.norm(S_q - S_fp)
