"""Asymmetric activation quantisation (Eq. 2-4) on the GPU against the oracle.

The GPU's codes, scales and zero points must be bit-exact with the
oracle's `quantize_rows_asym`, which is pinned by brute force in
test_oracle_pins. Its E4M3 operand carries two things:

- each code as an E4M3 byte, checked against the format's definition;
- 128 zero-point columns of E4M3(-z).

The weight rows carry 128 E4M3 values that must sum exactly to the row's
code sum. With both, the 4-bit GEMM over K + 128 must give
sum_k (q_a - z) q_w bit for bit, and the dequantised outputs must stay
within the usual tolerance.
"""

import numpy as np
import pytest
import torch

from oracle import sgat as osg
from paper_2606_04945_gb300 import inputs
from tests import helpers as H

pytestmark = pytest.mark.gpu


def unpack_unsigned(t):
    b = t.cpu().numpy().astype(np.int64)
    out = np.empty((b.shape[0], 2 * b.shape[1]), np.int64)
    out[:, 0::2] = b & 0xF
    out[:, 1::2] = b >> 4
    return out


def e4m3_value(b):
    """Value of E4M3 bytes (sign, 4 exponent bits with bias 7, 3 mantissa
    bits; normal numbers and the subnormal/zero exponent 0)."""
    b = np.asarray(b, np.int64)
    sign = np.where(b & 0x80, -1.0, 1.0)
    e = (b >> 3) & 0xF
    m = b & 7
    mag = np.where(e > 0, 2.0 ** (e - 7) * (1 + m / 8.0), 2.0 ** -6 * (m / 8.0))
    return sign * mag


def quant_asym(abi, X, mask, xf, with_xe=True):
    L, K = X.shape
    Xq = torch.empty(L, K // 2, dtype=torch.uint8, device="cuda")
    s_a = torch.empty(L, dtype=torch.float32, device="cuda")
    z_a = torch.empty(L, dtype=torch.int32, device="cuda")
    Xe = torch.empty(L, K + 128, dtype=torch.uint8, device="cuda") if with_xe else None
    abi.sgat_quantize_act_asym(X, mask, None if xf is None else H.dev(xf.a_m), None if xf is None else H.dev(xf.a_u),
                               xf.hb if xf else 1, xf.d_sh if xf else K, xf.d_m if xf else 0, xf.d_u if xf else 0,
                               Xq, s_a, z_a, Xe=Xe)
    abi.check_status()
    return Xq, s_a, z_a, Xe


@pytest.mark.parametrize("L,K,hb,dtype", [(37, 4096, 4096, "f16"), (130, 2048, 1024, "bf16"), (64, 512, 512, "f32"),
                                          (17, 256, 16, "f16"), (9, 1024, 64, "bf16")])
def test_quantize_act_asym_bitexact(abi, L, K, hb, dtype):
    case = inputs.random_linear(L + K + 3, L, K, 128, dtype=dtype, hb=hb)
    case.X[2] = 0                                               # an all-zero row
    xf = case.xf
    Xq, s_a, z_a, Xe = quant_asym(abi, H.dev(case.X, H.torch_dtype(dtype)), H.dev(case.mask), xf)
    codes, s, z = osg.sgat_quantize_act_asym(case.X, case.mask, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u)
    assert np.array_equal(unpack_unsigned(Xq), codes), "asymmetric codes differ"
    assert np.array_equal(s_a.cpu().numpy(), s), "scales differ"
    assert np.array_equal(z_a.cpu().numpy(), z), "zero points differ"
    assert s[2] == 0 and z[2] == 0
    xe = Xe.cpu().numpy()
    assert np.array_equal(xe[:, :K], H.e4m3_bytes(codes)), "E4M3 codes differ"
    assert np.array_equal(xe[:, K:], np.repeat(H.e4m3_bytes(-z)[:, None], 128, axis=1)), "zero-point columns differ"


def test_quantize_act_asym_positive_rows(abi):
    """Identity transform with every gate open and positive inputs: zero is
    the bottom of the range, so z = 0 and the codes span [0, 15]."""
    rng = np.random.default_rng(5)
    X = np.abs(rng.standard_normal((8, 256))).astype(np.float32)
    Xq, s_a, z_a, _ = quant_asym(abi, H.dev(X), None, None)
    codes, s, z = osg.sgat_quantize_act_asym(X, np.zeros(8, np.uint8), None, None, 1, 256, 0, 0)
    assert not z.any() and np.array_equal(z_a.cpu().numpy(), z)
    assert np.array_equal(unpack_unsigned(Xq), codes) and codes.max() == 15


@pytest.mark.parametrize("N,K", [(256, 4096), (96, 128), (64, 7680)])
def test_zero_point_columns(abi, N, K):
    """Weight rows: E4M3 codes, then 128 E4M3 values summing to the code sum
    (rows at the extremes: all +7 and all -7 reach |sum| = 7 K)."""
    rng = np.random.default_rng(N + K)
    q = rng.integers(-7, 8, (N, K))
    q[0] = 7
    q[1] = -7
    Wq = torch.from_numpy(osg.pack_int4(q)).cuda()
    We = torch.empty(N, K + 128, dtype=torch.uint8, device="cuda")
    abi.w4_zero_point_columns(Wq, We)
    abi.check_status()
    we = We.cpu().numpy()
    assert np.array_equal(we[:, :K], H.e4m3_bytes(q))
    sums = e4m3_value(we[:, K:]).sum(axis=1)
    assert np.array_equal(sums, q.sum(axis=1).astype(np.float64)), "zero-point columns do not sum to the code sums"


@pytest.mark.parametrize("L,K,N,hb,dtype", [(300, 4096, 384, 4096, "f16"), (64, 1024, 256, 512, "bf16"),
                                            (1024, 4096, 512, 4096, "f16"), (33, 256, 64, 16, "bf16")])
def test_sgat_linear_asym(abi, L, K, N, hb, dtype):
    """The fused asymmetric linear against the oracle's, and the GEMM over
    K + 128 bit for bit on the integer sums."""
    case = inputs.random_linear(L + N + 1, L, K, N, dtype=dtype, hb=hb, bias=True)
    xf = case.xf
    dt = H.torch_dtype(dtype)
    W = H.dev(case.W, dt)
    Wq = torch.empty(N, K // 2, dtype=torch.uint8, device="cuda")
    s_w = torch.empty(N, dtype=torch.float32, device="cuda")
    abi.sgat_prepare_weight(W, H.dev(xf.inv_a_w), hb, Wq, s_w)
    We = torch.empty(N, K + 128, dtype=torch.uint8, device="cuda")
    abi.w4_zero_point_columns(Wq, We)
    X = H.dev(case.X, dt)
    ws = torch.empty(abi.sgat_linear_asym_workspace_size(L, K), dtype=torch.uint8, device="cuda")
    Y = torch.empty(L, N, dtype=dt, device="cuda")
    abi.sgat_linear_asym(X, H.dev(case.mask), H.dev(xf.a_m), H.dev(xf.a_u), hb, xf.d_sh, xf.d_m, xf.d_u, We, s_w, Y,
                         ws, bias=H.dev(case.bias))
    abi.check_status()
    qw, sw_ref = osg.prepare_weight(case.W, xf.inv_a_w, hb, 4)
    Yr, codes, s, z, acc = osg.sgat_linear_asym(case.X, case.mask, xf.a_m, xf.a_u, hb, xf.d_sh, xf.d_m, xf.d_u, qw,
                                                sw_ref, bias=case.bias)
    a256 = lambda x: (x + 255) // 256 * 256
    o_s = a256(L * K // 2)
    o_e = o_s + 2 * a256(4 * L)
    assert np.array_equal(ws[o_s: o_s + 4 * L].view(torch.float32).cpu().numpy(), s)
    assert np.array_equal(ws[o_s + a256(4 * L): o_s + a256(4 * L) + 4 * L].view(torch.int32).cpu().numpy(), z)
    H.assert_output_close(H.host(Y), Yr, dtype)
    # the integer sums: the same operands through w4a4_gemm with acc_dbg
    Xe = ws[o_e: o_e + L * (K + 128)].view(L, K + 128)
    acc_g = torch.empty(L, N, dtype=torch.int32, device="cuda")
    Y2 = torch.empty(L, N, dtype=torch.float32, device="cuda")
    sa_t = ws[o_s: o_s + 4 * L].view(torch.float32)
    abi.w4a4_gemm(None, sa_t, None, s_w, Y2, acc_dbg=acc_g, Xe=Xe, We=We)
    abi.check_status()
    assert np.array_equal(acc_g.cpu().numpy().astype(np.int64), acc), "integer sums differ"
