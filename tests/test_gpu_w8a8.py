"""The 8-bit setting (W8A8, Tab. 5) on the GPU against the oracle.

The quantiser and the weight preparation take qmax = 127. Their codes and
scales must be bit-exact with the oracle (`oracle/sgat.py`, generic in the
bit width and pinned at 8 bits by brute force). The GEMM operand holds each
code as an fp16 number, checked against numpy's own float16 conversion of
the oracle's codes. w8a8_gemm's integer sums are compared bit for bit with
the oracle's exact integer product, and its outputs within the
dequantisation tolerance. This includes codes at ±127 everywhere, where
|acc| = 127² K exceeds the float32 integer range: only the int32 sum of the
kernel's 512-K runs (each below 2^23, exact in float32) reaches the full
value; K that is not a multiple of 512 (a short last run) and CTA pairs
that take several tiles (the run count carrying the accumulator parity
across tiles).
"""

import numpy as np
import pytest
import torch

from oracle import sgat as osg
from paper_2606_04945_gb300 import inputs
from tests import helpers as H

pytestmark = pytest.mark.gpu


def f16_bytes(codes):
    """Bytes [rows][2K] of 8-bit codes held as fp16 (little-endian halves)."""
    c = np.asarray(codes, dtype=np.int64)
    assert np.abs(c).max() <= 127
    return np.ascontiguousarray(c.astype(np.float16)).view(np.uint8)


def quant8(abi, case, with_xe=True):
    xf = case.xf
    X = H.dev(case.X, H.torch_dtype(case.dtype))
    L, K = case.X.shape
    Xq = torch.empty(L, K, dtype=torch.int8, device="cuda")
    s_a = torch.empty(L, dtype=torch.float32, device="cuda")
    Xe = torch.empty(L, 2 * K, dtype=torch.uint8, device="cuda") if with_xe else None
    abi.sgat_quantize_act(X, H.dev(case.mask), H.dev(xf.a_m), H.dev(xf.a_u), xf.hb, xf.d_sh, xf.d_m, xf.d_u,
                          Xq, s_a, bits=8, Xe=Xe)
    abi.check_status()
    return Xq, s_a, Xe


def prepare8(abi, case):
    N, K = case.W.shape
    Wq = torch.empty(N, K, dtype=torch.int8, device="cuda")
    s_w = torch.empty(N, dtype=torch.float32, device="cuda")
    abi.sgat_prepare_weight(H.dev(case.W, H.torch_dtype(case.dtype)), H.dev(case.xf.inv_a_w), case.xf.hb, Wq, s_w,
                            bits=8)
    We = torch.empty(N, 2 * K, dtype=torch.uint8, device="cuda")
    abi.w8_codes_f16(Wq, We)
    abi.check_status()
    return Wq, s_w, We


@pytest.mark.parametrize("L,K,hb,dtype", [(37, 4096, 4096, "f16"), (130, 2048, 1024, "bf16"), (64, 512, 512, "f32"),
                                          (17, 256, 16, "f16")])
def test_quantize_act_8bit_bitexact(abi, L, K, hb, dtype):
    case = inputs.random_linear(L + K + 8, L, K, 128, dtype=dtype, hb=hb)
    xf = case.xf
    Xq, s_a, Xe = quant8(abi, case)
    codes, s = osg.sgat_quantize_act(case.X, case.mask, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, 8)
    assert np.abs(codes).max() == 127                      # the row maxima reach qmax
    assert np.array_equal(Xq.cpu().numpy().astype(np.int64), codes), "8-bit codes differ"
    assert np.array_equal(s_a.cpu().numpy(), s), "scales differ"
    assert np.array_equal(Xe.cpu().numpy(), f16_bytes(codes)), "fp16 operand differs"


@pytest.mark.parametrize("N,K,hb,dtype", [(256, 4096, 4096, "bf16"), (128, 512, 512, "f16"), (384, 1024, 64, "f32")])
def test_prepare_weight_8bit_bitexact(abi, N, K, hb, dtype):
    case = inputs.random_linear(N + K, 16, K, N, dtype=dtype, hb=hb)
    Wq, s_w, We = prepare8(abi, case)
    q, s = osg.prepare_weight(case.W, case.xf.inv_a_w, hb, 8)
    assert np.array_equal(Wq.cpu().numpy().astype(np.int64), q), "8-bit weight codes differ"
    assert np.array_equal(s_w.cpu().numpy(), s)
    assert np.array_equal(We.cpu().numpy(), f16_bytes(q)), "fp16 operand differs"


def run_gemm(abi, qa, s_a, qw, s_w, y_dtype, bias=None):
    L, K = qa.shape
    N = qw.shape[0]
    Xe = torch.from_numpy(f16_bytes(qa)).cuda()
    Wq = torch.from_numpy(qw.astype(np.int8)).cuda()
    We = torch.empty(N, 2 * K, dtype=torch.uint8, device="cuda")
    abi.w8_codes_f16(Wq, We)
    assert np.array_equal(We.cpu().numpy(), f16_bytes(qw))
    Y = torch.empty(L, N, dtype=H.torch_dtype(y_dtype), device="cuda")
    acc = torch.empty(L, N, dtype=torch.int32, device="cuda")
    abi.w8a8_gemm(Xe, H.dev(s_a), We, H.dev(s_w), Y, bias=None if bias is None else H.dev(bias), acc_dbg=acc)
    abi.check_status()
    return H.host(Y), acc.cpu().numpy().astype(np.int64)


@pytest.mark.parametrize("L,N,K,y_dtype", [(128, 128, 128, "f32"), (200, 256, 4096, "f16"), (77, 384, 1024, "bf16"),
                                            (1, 128, 256, "f16"), (300, 640, 1152, "f16"), (513, 896, 2560, "bf16")])
def test_w8a8_gemm_matches_oracle(abi, L, N, K, y_dtype):
    """Random 8-bit codes over several tiles, a ragged last row tile and a
    ragged last column tile; K from one short run (128) to five runs with a
    short last one (2560 = 5 x 512; 1152 = 2 x 512 + 128)."""
    rng = np.random.default_rng(L * N + K)
    qa = rng.integers(-127, 128, (L, K))
    qw = rng.integers(-127, 128, (N, K))
    s_a = rng.uniform(0.001, 0.05, L).astype(np.float32)
    s_w = rng.uniform(0.001, 0.05, N).astype(np.float32)
    # no bias for float32 outputs: the helper's 1e-6 relative bound does not
    # cover the cancellation of a bias against the product
    bias = rng.normal(0, 0.1, N).astype(np.float32) if y_dtype != "f32" else None
    Y, acc = run_gemm(abi, qa, s_a, qw, s_w, y_dtype, bias)
    ref_acc = osg.int_gemm(qa, qw)
    assert np.array_equal(acc, ref_acc), "integer sums differ"
    H.assert_output_close(Y, osg.dequant(ref_acc, s_a, s_w, bias), y_dtype)


@pytest.mark.parametrize("pairs", [1, 2])
def test_w8a8_gemm_several_tiles_per_pair(abi, pairs):
    """Fewer CTA pairs than tiles (the pair limit): each pair runs several
    tiles, with three runs per tile (K = 1152), so that consecutive tiles
    start on alternate accumulators."""
    L, N, K = 300, 640, 1152                       # 2 x 3 tiles of 256 x 224
    rng = np.random.default_rng(pairs)
    qa = rng.integers(-127, 128, (L, K))
    qw = rng.integers(-127, 128, (N, K))
    s_a = rng.uniform(0.001, 0.05, L).astype(np.float32)
    s_w = rng.uniform(0.001, 0.05, N).astype(np.float32)
    bias = rng.normal(0, 0.1, N).astype(np.float32)
    prev = abi.set_gemm_pair_limit(pairs)
    try:
        Y, acc = run_gemm(abi, qa, s_a, qw, s_w, "f16", bias)
    finally:
        abi.set_gemm_pair_limit(prev)
    ref_acc = osg.int_gemm(qa, qw)
    assert np.array_equal(acc, ref_acc), "integer sums differ"
    H.assert_output_close(Y, osg.dequant(ref_acc, s_a, s_w, bias), "f16")


def test_w8a8_gemm_extreme_codes(abi):
    """Every code ±127 with aligned signs: |acc| = 127² K = 66 M at K = 4096,
    above 2^24. Each 512-K run's sum (127² 512 < 2^23) stays exact in
    float32 and only their int32 sum reaches the full value."""
    L, N, K = 128, 256, 4096
    rng = np.random.default_rng(1)
    sa = np.where(rng.random((L, 1)) < 0.5, -1, 1)
    sw = np.where(rng.random((N, 1)) < 0.5, -1, 1)
    qa = np.broadcast_to(sa * 127, (L, K)).copy()
    qw = np.broadcast_to(sw * 127, (N, K)).copy()
    s = np.full(L, 1e-6, np.float32)
    t = np.full(N, 1e-3, np.float32)
    Y, acc = run_gemm(abi, qa, s, qw, t, "f32")
    ref = osg.int_gemm(qa, qw)
    assert np.abs(ref).max() == 127 * 127 * K > 2 ** 24
    assert np.array_equal(acc, ref)
    H.assert_output_close(Y, osg.dequant(ref, s, t), "f32")


@pytest.mark.parametrize("L,K,N,hb,dtype,tac_g", [(300, 4096, 384, 4096, "f16", None), (64, 1024, 256, 512, "bf16", 64),
                                                  (1024, 4096, 512, 4096, "f16", 128)])
def test_sgat_linear_8bit(abi, L, K, N, hb, dtype, tac_g):
    """The fused 8-bit linear: codes (read back from the workspace) bit-exact
    with the oracle's on the same (TAC'd) input, integer sums exact (checked
    through w8a8_gemm on the same codes), outputs within tolerance."""
    case = inputs.random_linear(L + N, L, K, N, dtype=dtype, hb=hb, tac_g=tac_g, bias=True)
    xf = case.xf
    Wq, s_w, We = prepare8(abi, case)
    dt = H.torch_dtype(dtype)
    X = H.dev(case.X, dt)
    ws = torch.empty(abi.sgat_linear_workspace_size(L, K, tac_g is not None, bits=8), dtype=torch.uint8,
                     device="cuda")
    Y = torch.empty(L, N, dtype=dt, device="cuda")
    tac_M = H.dev(case.tac.M) if tac_g else None
    tac_d = H.dev(case.tac.d) if tac_g else None
    abi.sgat_linear(X, H.dev(case.mask), H.dev(xf.a_m), H.dev(xf.a_u), xf.hb, xf.d_sh, xf.d_m, xf.d_u, None, s_w, Y,
                    ws, bias=H.dev(case.bias), tac_M=tac_M, tac_d=tac_d, tac_g=tac_g or 0, bits=8, We=We)
    abi.check_status()
    a256 = lambda x: (x + 255) // 256 * 256
    # [code region, left unwritten][s_a][Xe: each code as fp16]
    s_a = ws[a256(L * K): a256(L * K) + 4 * L].view(torch.float32).cpu().numpy()
    o_e = a256(L * K) + a256(4 * L)
    Xe = ws[o_e: o_e + 2 * L * K].cpu().numpy()
    Xq = Xe.view(np.float16).reshape(L, K).astype(np.int64)
    assert np.array_equal(f16_bytes(Xq), Xe.reshape(L, 2 * K)), "operand bytes are not fp16 integers"
    if tac_g:
        o = a256(L * K) + a256(4 * L) + a256(2 * L * K)
        esz = torch.empty(0, dtype=dt).element_size()
        qin = ws[o: o + esz * L * K].view(dt).view(L, K).float().cpu().numpy()     # the GPU's TAC output
    else:
        qin = case.X.astype(np.float32)
    codes, s = osg.sgat_quantize_act(qin, case.mask, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, 8)
    assert np.array_equal(Xq, codes), "8-bit codes differ"
    assert np.array_equal(s_a, s), "scales differ"
    qw, sw_ref = osg.prepare_weight(case.W, xf.inv_a_w, hb, 8)
    rows = np.arange(L) if L <= 300 else np.random.default_rng(0).choice(L, 96, replace=False)
    ref_acc = osg.int_gemm(codes[rows], qw)
    ref = osg.dequant(ref_acc, s[rows], sw_ref, case.bias)
    H.assert_output_close(H.host(Y)[rows], ref, dtype)


def test_w8a8_empty_batch(abi):
    """L = 0 (N = 0 for the weight form) is a valid no-op of every 8-bit
    entry point."""
    K, N = 512, 256
    X = torch.empty(0, K, dtype=torch.float16, device="cuda")
    Xq = torch.empty(0, K, dtype=torch.int8, device="cuda")
    s = torch.empty(0, dtype=torch.float32, device="cuda")
    Xe = torch.empty(0, 2 * K, dtype=torch.uint8, device="cuda")
    abi.sgat_quantize_act(X, None, None, None, 512, K, 0, 0, Xq, s, bits=8, Xe=Xe)
    We = torch.zeros(N, 2 * K, dtype=torch.uint8, device="cuda")
    sw = torch.ones(N, dtype=torch.float32, device="cuda")
    Y = torch.empty(0, N, dtype=torch.float16, device="cuda")
    abi.w8a8_gemm(Xe, s, We, sw, Y)
    abi.w8_codes_f16(torch.empty(0, K, dtype=torch.int8, device="cuda"),
                     torch.empty(0, 2 * K, dtype=torch.uint8, device="cuda"))
    ws = torch.empty(256, dtype=torch.uint8, device="cuda")
    abi.sgat_linear(X, None, None, None, 512, K, 0, 0, None, sw, Y, ws, bits=8, We=We)
    abi.check_status()
