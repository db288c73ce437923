"""The dense orthogonal basis (the learned P of App. B) on the GPU against
the oracle.

The transform X^s P runs on the 16-bit GEMM. Its operands are float16 and
its result is stored as float16. The GPU's V therefore may differ from the
oracle's (a float64 product rounded once) where the float32 accumulation
error moves the sum across a float16 rounding boundary. That is a few
steps at most, where the sum cancels. The checks:

- V agrees with the oracle within the float32 accumulation bound plus one
  float16 spacing, and exactly at most places;
- the codes and scales are bit-exact with the oracle's quantiser applied to
  the GPU's own V (teacher forcing), on both the activation and the weight
  side;
- the linear's outputs are within tolerance of the dequantised exact
  integer product of those codes, and close to the oracle's own dense
  linear.

P is orthogonal: the QR factor of a Gaussian matrix, rounded to float16.
"""

import numpy as np
import pytest
import torch

from oracle import sgat as osg
from paper_2606_04945_gb300 import inputs
from tests import helpers as H

pytestmark = pytest.mark.gpu


def basis(K, seed):
    Q, _ = np.linalg.qr(np.random.default_rng(seed).standard_normal((K, K)))
    P = Q.astype(np.float16)
    return P, torch.from_numpy(np.ascontiguousarray(P.T)).cuda()


def check_v(v_gpu, v_ref, A, P):
    """The GPU's float32 accumulation of the float16 product differs from the
    exact sum by at most K u sum_k |a_k p_k| (u = 2^-24; a factor 8 of
    margin for the tensor cores' accumulation order), plus one float16
    rounding of the result."""
    a16 = np.abs(np.asarray(A, np.float32).astype(np.float16).astype(np.float64))
    bound = 8 * a16.shape[1] * 2.0 ** -24 * (a16 @ np.abs(P.astype(np.float64)))
    spacing = np.spacing(np.abs(v_ref).astype(np.float16)).astype(np.float64)
    assert np.all(np.abs(v_gpu.astype(np.float64) - v_ref) <= spacing + bound), "V outside the accumulation bound"
    assert np.mean(v_gpu == v_ref) > 0.95, "V differs from the oracle too often"


def gated(V, mask, d_sh, d_m, d_u):
    K = V.shape[1]
    g_m, g_u = osg.state_gates(K, d_sh, d_m, d_u)
    g = np.where(np.asarray(mask)[:, None] != 0, g_m[None, :], g_u[None, :])
    return np.where(g != 0, V, np.float32(0)).astype(np.float32)


@pytest.mark.parametrize("L,K,dtype", [(64, 512, "f16"), (130, 1024, "bf16"), (33, 4096, "f32")])
def test_quantize_act_dense(abi, L, K, dtype):
    case = inputs.random_linear(L + K + 5, L, K, 128, dtype=dtype, hb=1)
    xf = case.xf
    P, Pt = basis(K, K)
    Xq = torch.empty(L, K // 2, dtype=torch.uint8, device="cuda")
    s_a = torch.empty(L, dtype=torch.float32, device="cuda")
    Xe = torch.empty(L, K, dtype=torch.uint8, device="cuda")
    ws = abi.sgat_quantize_act_dense(H.dev(case.X, H.torch_dtype(dtype)), H.dev(case.mask), H.dev(xf.a_m),
                                     H.dev(xf.a_u), Pt, xf.d_sh, xf.d_m, xf.d_u, Xq, s_a, Xe=Xe)
    abi.check_status()
    o = (L * K * 2 + 255) // 256 * 256
    v_gpu = ws[o: o + 2 * L * K].view(torch.float16).view(L, K).float().cpu().numpy()
    codes_ref, s_ref, v_ref = osg.sgat_quantize_act_dense(case.X, case.mask, xf.a_m, xf.a_u, P, xf.d_sh, xf.d_m,
                                                          xf.d_u)
    a_rows = np.where(case.mask[:, None] != 0, xf.a_m[None, :], xf.a_u[None, :]).astype(np.float32)
    check_v(v_gpu, v_ref, (case.X.astype(np.float32) * a_rows).astype(np.float32), P)
    q, s = osg.quantize_rows_sym(gated(v_gpu, case.mask, xf.d_sh, xf.d_m, xf.d_u), 4)
    assert np.array_equal(H.unpack(Xq), q), "codes differ from the oracle's on the GPU's V"
    assert np.array_equal(s_a.cpu().numpy(), s)
    assert np.array_equal(Xe.cpu().numpy(), H.e4m3_bytes(q))
    flips = H.unpack(Xq) != codes_ref
    assert flips.mean() < 0.02 and np.all(np.abs(H.unpack(Xq) - codes_ref)[flips] == 1)


@pytest.mark.parametrize("N,K,dtype", [(256, 1024, "f16"), (128, 4096, "bf16")])
def test_prepare_weight_dense(abi, N, K, dtype):
    case = inputs.random_linear(N + K, 8, K, N, dtype=dtype, hb=1)
    P, Pt = basis(K, K + 1)
    Wq = torch.empty(N, K // 2, dtype=torch.uint8, device="cuda")
    s_w = torch.empty(N, dtype=torch.float32, device="cuda")
    ws = abi.sgat_prepare_weight_dense(H.dev(case.W, H.torch_dtype(dtype)), H.dev(case.xf.inv_a_w), Pt, Wq, s_w)
    abi.check_status()
    o = (N * K * 2 + 255) // 256 * 256
    wf_gpu = ws[o: o + 2 * N * K].view(torch.float16).view(N, K).float().cpu().numpy()
    _, _, wf_ref = osg.prepare_weight_dense(case.W, case.xf.inv_a_w, P)
    check_v(wf_gpu, wf_ref, (case.W.astype(np.float32) * case.xf.inv_a_w[None, :]).astype(np.float32), P)
    q, s = osg.quantize_rows_sym(wf_gpu, 4)
    assert np.array_equal(H.unpack(Wq), q) and np.array_equal(s_w.cpu().numpy(), s)


@pytest.mark.parametrize("L,K,N,dtype", [(200, 1024, 256, "f16"), (1024, 4096, 384, "f16")])
def test_sgat_linear_dense(abi, L, K, N, dtype):
    case = inputs.random_linear(L + N + 2, L, K, N, dtype=dtype, hb=1, bias=True)
    xf = case.xf
    P, Pt = basis(K, L + K)
    dt = H.torch_dtype(dtype)
    Wq = torch.empty(N, K // 2, dtype=torch.uint8, device="cuda")
    s_w = torch.empty(N, dtype=torch.float32, device="cuda")
    abi.sgat_prepare_weight_dense(H.dev(case.W, dt), H.dev(xf.inv_a_w), Pt, Wq, s_w)
    We = torch.empty(N, K, dtype=torch.uint8, device="cuda")
    abi.w4_unpack_e4m3(Wq, We)
    ws = torch.empty(abi.sgat_linear_dense_workspace_size(L, K), dtype=torch.uint8, device="cuda")
    Y = torch.empty(L, N, dtype=dt, device="cuda")
    abi.sgat_linear_dense(H.dev(case.X, dt), H.dev(case.mask), H.dev(xf.a_m), H.dev(xf.a_u), Pt, xf.d_sh, xf.d_m,
                          xf.d_u, Wq, s_w, Y, ws, bias=H.dev(case.bias), We=We)
    abi.check_status()
    a256 = lambda x: (x + 255) // 256 * 256
    o = 2 * a256(2 * L * K)                       # then [packed-code region, unwritten][s_a][Xe]
    o_e = o + a256(L * K // 2) + a256(4 * L)
    codes = H.codes_from_e4m3(ws[o_e: o_e + L * K].view(L, K))
    s_a = ws[o + a256(L * K // 2): o + a256(L * K // 2) + 4 * L].view(torch.float32).cpu().numpy()
    qw, sw = H.unpack(Wq), s_w.cpu().numpy()
    ref = osg.dequant(osg.int_gemm(codes, qw), s_a, sw, case.bias)
    H.assert_output_close(H.host(Y), ref, dtype)
    # end to end against the oracle's own dense linear (no teacher forcing):
    # codes that flip at rounding boundaries move the outputs only slightly
    codes_o, s_o, _ = osg.sgat_quantize_act_dense(case.X, case.mask, xf.a_m, xf.a_u, P, xf.d_sh, xf.d_m, xf.d_u)
    qw_o, sw_o, _ = osg.prepare_weight_dense(case.W, xf.inv_a_w, P)
    Y_o = osg.dequant(osg.int_gemm(codes_o, qw_o), s_o, sw_o, case.bias)
    assert np.linalg.norm(H.host(Y) - Y_o) / np.linalg.norm(Y_o) < 0.02


def test_sgat_linear_dense_calibrated_basis(abi):
    """The dense path on a basis calibrated by App. B's procedure (the
    oracle's AdamW calibration on the Eq. 15 objective, paper settings, on
    a synthetic calibration set): the GPU's codes and outputs match the
    oracle on that basis (teacher-forced, as above), and the calibrated
    basis gives a smaller error against the full-precision product X W^T
    than the orthogonalised Gaussian it started from."""
    from oracle import calibration as oc
    K = N = 256
    d_m = d_u = K // 32
    d_sh = K - 2 * d_m
    samples, W = inputs.basis_calibration_set(21, K, n_samples=8, tokens=64, N=N)
    P_cal, hist = oc.calibrate_basis(samples, W, d_sh, d_m, d_u, seed=3)
    assert hist["objective"][-1] < hist["objective"][0]
    X, mask = inputs.basis_calibration_set(22, K, n_samples=1, tokens=200, N=N)[0][0]
    X16 = X.astype(np.float16)
    ones = np.ones(K, np.float32)
    errs = []
    for P in (oc.orthogonal_init(K, 3), P_cal):
        P16 = P.astype(np.float16)
        Pt = torch.from_numpy(np.ascontiguousarray(P16.T)).cuda()
        Wq = torch.empty(N, K // 2, dtype=torch.uint8, device="cuda")
        s_w = torch.empty(N, dtype=torch.float32, device="cuda")
        abi.sgat_prepare_weight_dense(H.dev(W, torch.float16), H.dev(ones), Pt, Wq, s_w)
        We = torch.empty(N, K, dtype=torch.uint8, device="cuda")
        abi.w4_unpack_e4m3(Wq, We)
        L = X.shape[0]
        ws = torch.empty(abi.sgat_linear_dense_workspace_size(L, K), dtype=torch.uint8, device="cuda")
        Y = torch.empty(L, N, dtype=torch.float16, device="cuda")
        abi.sgat_linear_dense(H.dev(X16, torch.float16), H.dev(mask), H.dev(ones), H.dev(ones), Pt, d_sh, d_m, d_u,
                              Wq, s_w, Y, ws, We=We)
        abi.check_status()
        a256 = lambda x: (x + 255) // 256 * 256
        o = 2 * a256(2 * L * K)                   # then [packed-code region, unwritten][s_a][Xe]
        o_e = o + a256(L * K // 2) + a256(4 * L)
        codes = H.codes_from_e4m3(ws[o_e: o_e + L * K].view(L, K))
        s_a = ws[o + a256(L * K // 2): o + a256(L * K // 2) + 4 * L].view(torch.float32).cpu().numpy()
        v_gpu = ws[a256(2 * L * K): a256(2 * L * K) + 2 * L * K].view(torch.float16).view(L, K).float().cpu().numpy()
        q, s = osg.quantize_rows_sym(gated(v_gpu, mask, d_sh, d_m, d_u), 4)
        assert np.array_equal(codes, q) and np.array_equal(s_a, s), "codes on the GPU's V"
        ref = osg.dequant(osg.int_gemm(codes, H.unpack(Wq)), s_a, s_w.cpu().numpy(), None)
        H.assert_output_close(H.host(Y), ref, "f16")
        exact = X16.astype(np.float64) @ W.astype(np.float64).T
        errs.append(np.linalg.norm(H.host(Y) - exact) / np.linalg.norm(exact))
    assert errs[1] < errs[0], errs
