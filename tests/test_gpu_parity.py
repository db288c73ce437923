"""GPU (libstarq.so through its C ABI) against the CPU oracle.

Bit-exact: packed int4 codes, per-row scales, float32 transformed values and
the integer accumulators. Tolerance (tests/helpers.py): dequantised outputs
and TAC. Sizes run from one token to several tiles with ragged tails, plus
the edge cases of the method (all-zero rows, all-masked / all-unmasked
batches, no mask, identity transform, gates off).
"""

import numpy as np
import pytest
import torch

from oracle import sgat as osg
from oracle import tac as otac
from paper_2606_04945_gb300 import inputs
from tests import helpers as H

pytestmark = pytest.mark.gpu


def run_quant(abi, case, mask=True, dbg=True):
    xf = case.xf
    X = H.dev(case.X, H.torch_dtype(case.dtype))
    L, K = case.X.shape
    m = H.dev(case.mask) if mask else None
    a_m, a_u = H.dev(xf.a_m), H.dev(xf.a_u)
    Xq = torch.empty(L, K // 2, dtype=torch.uint8, device="cuda")
    s_a = torch.empty(L, dtype=torch.float32, device="cuda")
    Xe = torch.empty(L, K, dtype=torch.uint8, device="cuda")
    v = torch.empty(L, K, dtype=torch.float32, device="cuda") if dbg else None
    abi.sgat_quantize_act(X, m, a_m, a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, Xq, s_a, Xe=Xe, v_dbg=v)
    abi.check_status()
    assert np.array_equal(Xe.cpu().numpy(), H.e4m3_bytes(H.unpack(Xq))), "E4M3 copy differs from the codes"
    return Xq, s_a, v


QUANT_CASES = [
    # (L, K, hb, dtype, gates_on)
    (1, 512, 512, "f16", True),
    (7, 128, 128, "f16", True),
    (33, 3584, 512, "bf16", True),
    (129, 4096, 4096, "f16", True),
    (5, 12288, 4096, "f16", True),
    (3, 18944, 512, "bf16", True),
    (64, 1024, 1024, "f16", False),
    (40, 2048, 2048, "f32", True),
    (9, 256, 16, "f16", True),
    (9, 256, 1, "f16", False),
    (300, 640, 128, "f16", True),
    # rows of 1024-or-larger blocks: one CTA per row, rounds of 4096 features
    (17, 8192, 2048, "bf16", True),       # two rounds
    (6, 16384, 4096, "f16", True),        # four rounds
    (11, 5120, 1024, "f32", True),        # last round holds one chunk
    (4, 6144, 2048, "f16", False),        # last round holds one 2048 block
    (3, 20480, 4096, "f16", True),        # beyond 16384 features: warp-per-chunk kernel
    # warp-per-chunk rows: a half last 1024-chunk, small blocks, 20 warps per row
    (20, 1536, 64, "f32", True),
    (13, 2560, 1, "f16", False),
    (7, 20480, 512, "bf16", True),
]


@pytest.mark.parametrize("L,K,hb,dtype,gates", QUANT_CASES)
def test_quantize_act_bitexact(abi, L, K, hb, dtype, gates):
    case = inputs.random_linear(L + K + hb, L, K, 128, dtype=dtype, gates_on=gates, hb=hb)
    xf = case.xf
    Xq, s_a, v = run_quant(abi, case)
    codes, s = osg.sgat_quantize_act(case.X, case.mask, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, 4)
    V = osg.sgat_transform(case.X, case.mask, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u)
    assert np.array_equal(v.cpu().numpy(), V), "transformed activations differ"
    assert np.array_equal(H.unpack(Xq), codes), "int4 codes differ"
    assert np.array_equal(s_a.cpu().numpy(), s), "scales differ"


@pytest.mark.parametrize("L,K,hb,dtype,bits", [(129, 4096, 4096, "f16", 4), (33, 3584, 512, "bf16", 4),
                                                (9, 256, 16, "f16", 4), (40, 2048, 2048, "f32", 8)])
def test_quantize_act_without_packed_codes(abi, L, K, hb, dtype, bits):
    """Xq = NULL with Xe given (the form sgat_linear and the grouped step
    use): the operand bytes and scales equal those of a call that also
    writes the packed codes (row kernel, warp-per-chunk kernel, 8-bit)."""
    case = inputs.random_linear(L + K + hb + bits, L, K, 128, dtype=dtype, gates_on=True, hb=hb)
    xf = case.xf
    X, m = H.dev(case.X, H.torch_dtype(dtype)), H.dev(case.mask)
    a_m, a_u = H.dev(xf.a_m), H.dev(xf.a_u)
    qb = K // 2 if bits == 4 else K
    eb = K if bits == 4 else 2 * K
    Xq = torch.empty(L, qb, dtype=torch.uint8, device="cuda")
    s1, s2 = (torch.empty(L, dtype=torch.float32, device="cuda") for _ in range(2))
    Xe1, Xe2 = (torch.empty(L, eb, dtype=torch.uint8, device="cuda") for _ in range(2))
    abi.sgat_quantize_act(X, m, a_m, a_u, hb, xf.d_sh, xf.d_m, xf.d_u, Xq, s1, bits=bits, Xe=Xe1)
    abi.sgat_quantize_act(X, m, a_m, a_u, hb, xf.d_sh, xf.d_m, xf.d_u, None, s2, bits=bits, Xe=Xe2)
    abi.check_status()
    assert torch.equal(Xe1, Xe2) and torch.equal(s1, s2)


@pytest.mark.parametrize("L,K,hb,dtype", [(300, 4096, 4096, "f16"), (77, 1024, 512, "bf16"), (5, 2048, 2048, "f32"),
                                           (1, 3584, 512, "bf16"), (9, 12288, 4096, "f16"), (4, 256, 16, "f16")])
def test_quantize_act_grouped(abi, L, K, hb, dtype):
    """Two quantisations in one launch (each problem with its own input,
    mask, smoothing vectors and gate layout): both against the oracle (codes
    and scales bit for bit), and bit-identical to two single calls. The
    last two shapes (rows beyond 4096 features, blocks of 16) fall back to
    two launches."""
    cases = [inputs.random_linear(L + K + hb + 11 * t, L, K, 128, dtype=dtype, gates_on=(t == 0), hb=hb)
             for t in range(2)]
    td = H.torch_dtype(dtype)
    ios, outs = [], []
    for c in cases:
        xf = c.xf
        io = dict(X=H.dev(c.X, td), mask=H.dev(c.mask), a_m=H.dev(xf.a_m), a_u=H.dev(xf.a_u), d_sh=xf.d_sh,
                  d_m=xf.d_m, d_u=xf.d_u, Xq=torch.empty(L, K // 2, dtype=torch.uint8, device="cuda"),
                  s_a=torch.empty(L, dtype=torch.float32, device="cuda"),
                  Xe=torch.empty(L, K, dtype=torch.uint8, device="cuda"))
        ios.append(io)
    abi.sgat_quantize_act_grouped(ios[0], ios[1], hb)
    abi.check_status()
    for c, io in zip(cases, ios):
        xf = c.xf
        codes, sc = osg.sgat_quantize_act(c.X, c.mask, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, 4)
        assert np.array_equal(H.unpack(io["Xq"]), codes), "int4 codes differ"
        assert np.array_equal(io["s_a"].cpu().numpy(), sc), "scales differ"
        assert np.array_equal(io["Xe"].cpu().numpy(), H.e4m3_bytes(codes)), "E4M3 codes differ"
        Xq1, s1, Xe1 = torch.empty_like(io["Xq"]), torch.empty_like(io["s_a"]), torch.empty_like(io["Xe"])
        abi.sgat_quantize_act(io["X"], io["mask"], io["a_m"], io["a_u"], hb, io["d_sh"], io["d_m"], io["d_u"], Xq1,
                              s1, Xe=Xe1)
        abi.check_status()
        assert torch.equal(Xq1, io["Xq"]) and torch.equal(s1, io["s_a"]) and torch.equal(Xe1, io["Xe"])


@pytest.mark.parametrize("K,hb", [(4096, 4096), (2048, 1024), (1024, 512), (256, 16)])
def test_quantize_act_exact_ties(abi, K, hb):
    """Transformed values that sit exactly on a rounding tie (x.5 after the
    scaling by r = 7 / amax, an exact power of two here): the codes round
    half to even. X = v H / hb per block is exact in float32, and the
    float32 butterflies of X reproduce v exactly (dyadic partial sums)."""
    rng = np.random.default_rng(K + hb)
    L = 12
    V = np.zeros((L, K))
    ties = np.array([0.5, 1.5, 2.5, 3.5, 4.5, 5.5, 6.5])
    for i in range(L):
        scale = 2.0 ** (i - 4)                       # amax = 7 * scale, r = 1 / scale
        pos = rng.choice(K, 2 * len(ties) + 1, replace=False)
        V[i, pos[0]] = 7 * scale * (-1) ** i
        V[i, pos[1:1 + len(ties)]] = ties * scale
        V[i, pos[1 + len(ties):]] = -ties * scale
    Hh = osg.hadamard_sylvester(hb).astype(np.float64)
    X = (V.reshape(L, K // hb, hb) @ Hh / hb).reshape(L, K).astype(np.float32)
    Xq = torch.empty(L, K // 2, dtype=torch.uint8, device="cuda")
    s_a = torch.empty(L, dtype=torch.float32, device="cuda")
    Xe = torch.empty(L, K, dtype=torch.uint8, device="cuda")
    abi.sgat_quantize_act(H.dev(X), None, None, None, hb, K, 0, 0, Xq, s_a, Xe=Xe)
    abi.check_status()
    codes, s = osg.sgat_quantize_act(X, np.zeros(L, np.uint8), None, None, hb, K, 0, 0, 4)
    nz = V != 0
    expect = np.where(np.abs(V / (np.abs(V).max(1, keepdims=True) / 7)) % 1 == 0.5, 0, 1)
    assert (nz & (expect == 0)).sum() == L * 2 * len(ties)          # the ties are there
    assert np.array_equal(codes[nz], np.rint(V[nz] / (np.abs(V).max(1, keepdims=True) / 7).repeat(K, 1)[nz]))
    assert np.array_equal(H.unpack(Xq), codes), "codes at exact ties differ"
    assert np.array_equal(s_a.cpu().numpy(), s)
    assert np.array_equal(Xe.cpu().numpy(), H.e4m3_bytes(codes))


@pytest.mark.parametrize("K,hb", [(512, 512), (4096, 4096)])
def test_quantize_act_edge_cases(abi, K, hb):
    """No mask (all unmasked), all masked, mixed; an all-zero row in each."""
    case = inputs.random_linear(5, 24, K, 128, hb=hb)
    case.X[3] = 0
    xf = case.xf
    mixed = case.mask.copy()
    for mode in ("none", "all", "mixed"):
        if mode == "none":
            mask_np = np.zeros(case.L, np.uint8)
            Xq, s_a, _ = run_quant(abi, case, mask=False)
        else:
            mask_np = np.ones(case.L, np.uint8) if mode == "all" else mixed
            case.mask = mask_np
            Xq, s_a, _ = run_quant(abi, case)
        codes, s = osg.sgat_quantize_act(case.X, mask_np, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, 4)
        assert np.array_equal(H.unpack(Xq), codes), mode
        assert np.array_equal(s_a.cpu().numpy(), s), mode
        assert s[3] == 0 and not codes[3].any()


@pytest.mark.parametrize("N,K,hb,dtype", [(256, 512, 512, "f16"), (96, 4096, 4096, "bf16"),
                                          (64, 18944, 512, "bf16"), (32, 128, 1, "f32")])
def test_prepare_weight_bitexact(abi, N, K, hb, dtype):
    case = inputs.random_linear(N + K, 16, K, N, dtype=dtype, hb=hb)
    W = H.dev(case.W, H.torch_dtype(dtype))
    inv = H.dev(case.xf.inv_a_w)
    Wq = torch.empty(N, K // 2, dtype=torch.uint8, device="cuda")
    s_w = torch.empty(N, dtype=torch.float32, device="cuda")
    abi.sgat_prepare_weight(W, inv, hb, Wq, s_w)
    abi.check_status()
    q, s = osg.prepare_weight(case.W, case.xf.inv_a_w, hb, 4)
    assert np.array_equal(H.unpack(Wq), q)
    assert np.array_equal(s_w.cpu().numpy(), s)


def unpacked_weight(abi, Wq):
    """The E4M3 weight bytes of packed codes, by w4_unpack_e4m3."""
    We = torch.empty(Wq.shape[0], 2 * Wq.shape[1], dtype=torch.uint8, device="cuda")
    abi.w4_unpack_e4m3(Wq, We)
    return We


def run_gemm(abi, qa, qw, s_a, s_w, out="f16", bias=None, path="e4m3"):
    """path "packed": packed int4 activations (both operands converted in the
    kernel); "e4m3": E4M3 activation codes by TMA to CTA pairs that convert
    the weights; "tma": both operands as E4M3 bytes by TMA (weights unpacked
    by w4_unpack_e4m3, checked against the format's definition)."""
    L, K = qa.shape
    N = qw.shape[0]
    Wq = H.dev(osg.pack_int4(qw))
    Y = torch.empty(L, N, dtype=H.torch_dtype(out), device="cuda")
    acc = torch.empty(L, N, dtype=torch.int32, device="cuda")
    We = None
    if path == "packed":
        Xq, Xe = H.dev(osg.pack_int4(qa)), None
    else:
        Xq, Xe = None, H.dev(H.e4m3_bytes(qa))
    if path == "tma":
        We = unpacked_weight(abi, Wq)
        assert np.array_equal(We.cpu().numpy(), H.e4m3_bytes(qw)), "unpacked weight bytes differ"
        Wq = None
    abi.w4a4_gemm(Xq, H.dev(s_a), Wq, H.dev(s_w), Y, bias=None if bias is None else H.dev(bias),
                  acc_dbg=acc, Xe=Xe, We=We)
    abi.check_status()
    return H.host(Y), acc.cpu().numpy()


@pytest.mark.parametrize("N,K", [(1, 32), (3, 96), (1000, 4096), (4096, 64)])
def test_w4_unpack_e4m3(abi, N, K):
    """Every byte value of the packed codes (both nibbles, -8 included) maps
    to the E4M3 byte of its integer."""
    rng = np.random.default_rng(N * 7 + K)
    packed = rng.integers(0, 256, (N, K // 2), dtype=np.uint8)
    flat = packed.reshape(-1)
    flat[: min(256, flat.size)] = np.arange(min(256, flat.size), dtype=np.uint8)
    We = unpacked_weight(abi, H.dev(packed))
    abi.check_status()
    assert np.array_equal(We.cpu().numpy(), H.e4m3_bytes(osg.unpack_int4(packed)))


@pytest.mark.parametrize("path", ["tma", "e4m3", "packed"])
@pytest.mark.parametrize("L,N,K,out", [(1, 256, 128, "f16"), (129, 512, 512, "f16"), (300, 288, 1024, "bf16"),
                                       (128, 256, 4096, "f32"), (1000, 768, 384, "f16"),
                                       (257, 4096, 256, "f16"), (513, 160, 640, "f16")])
def test_w4a4_gemm_exact(abi, L, N, K, out, path):
    qa, qw, s_a, s_w = H.gemm_codes(L * 7 + N + K, L, N, K)
    bias = np.random.default_rng(1).normal(0, 0.1, N).astype(np.float32) if out == "bf16" else None
    Y, acc = run_gemm(abi, qa, qw, s_a, s_w, out, bias, path)
    ref_acc = osg.int_gemm(qa, qw)
    assert np.array_equal(acc, ref_acc), "integer accumulators differ"
    H.assert_output_close(Y, osg.dequant(ref_acc, s_a, s_w, bias), out)


@pytest.mark.parametrize("out", ["f16", "f32"])
def test_w4a4_gemm_tile_widths(abi, out):
    """The launcher takes 256-channel pair tiles (two pairs per cluster) or
    224-channel tiles on single pairs, whichever its estimate makes cheaper.
    4608 x 1024 fills 36 clusters exactly with 256-wide tiles (224 would need
    a second round); 97 x 256 is one round either way, and the narrower tile
    has the cheaper stage; the LLaDA widths 4096 and 12288 (at a short K)
    favour 224. Every product is exact, and both widths occur."""
    seen = set()
    for L, N, K in [(4608, 1024, 128), (97, 256, 128), (1024, 4096, 256), (1024, 12288, 256), (300, 4128, 384)]:
        qa, qw, s_a, s_w = H.gemm_codes(L + N + K, L, N, K)
        Y, acc = run_gemm(abi, qa, qw, s_a, s_w, out, path="tma")
        bn, cl = abi.last_gemm_tile()
        seen.add(bn)
        ref = osg.int_gemm(qa, qw)
        assert np.array_equal(acc, ref), f"integer accumulators differ ({L}x{N}x{K}, tile {bn}/{cl})"
        H.assert_output_close(Y, osg.dequant(ref, s_a, s_w, None), out)
    assert seen == {224, 256}, seen


@pytest.mark.parametrize("L,N0,N1,K,out", [(300, 768, 288, 512, "f16"), (1, 256, 32, 128, "bf16"),
                                            (513, 160, 4096, 256, "f32"), (257, 4096, 12288, 128, "f16")])
def test_w4a4_gemm_grouped(abi, L, N0, N1, K, out):
    """Two products in one launch (problem 1's tiles follow problem 0's):
    the exact integer sums of both against the oracle, outputs within the
    dequantisation bound, and each bit-identical to a w4a4_gemm call of its
    own. Ragged L, widths that are not multiples of the pair tile, a bias
    on one problem only, and more tiles than CTA pairs (257 x 16384)."""
    qa0, qw0, s_a0, s_w0 = H.gemm_codes(L + N0 + K, L, N0, K)
    qa1, qw1, s_a1, s_w1 = H.gemm_codes(L + N1 + 2 * K + 1, L, N1, K)
    bias1 = np.random.default_rng(L + 5).normal(0, 0.1, N1).astype(np.float32)
    Xe0, Xe1 = H.dev(H.e4m3_bytes(qa0)), H.dev(H.e4m3_bytes(qa1))
    We0, We1 = H.dev(H.e4m3_bytes(qw0)), H.dev(H.e4m3_bytes(qw1))
    sa0, sa1, sw0, sw1, b1 = H.dev(s_a0), H.dev(s_a1), H.dev(s_w0), H.dev(s_w1), H.dev(bias1)
    td = H.torch_dtype(out)
    Y0 = torch.empty(L, N0, dtype=td, device="cuda")
    Y1 = torch.empty(L, N1, dtype=td, device="cuda")
    acc0 = torch.empty(L, N0, dtype=torch.int32, device="cuda")
    acc1 = torch.empty(L, N1, dtype=torch.int32, device="cuda")
    abi.w4a4_gemm_grouped(Xe0, sa0, We0, sw0, Y0, Xe1, sa1, We1, sw1, Y1, bias1=b1, acc_dbg0=acc0, acc_dbg1=acc1,
                          weights_ready=(L == 300))
    abi.check_status()
    ref0, ref1 = osg.int_gemm(qa0, qw0), osg.int_gemm(qa1, qw1)
    assert np.array_equal(acc0.cpu().numpy(), ref0), "integer accumulators differ (problem 0)"
    assert np.array_equal(acc1.cpu().numpy(), ref1), "integer accumulators differ (problem 1)"
    if out == "f32":
        # float32 output: Eq. 3's float32 steps, each rounded (a bias can
        # cancel most of the product, so a float64 reference with a relative
        # bound would not fit): bit for bit
        def deq32(acc, sa, sw, b):
            y = (acc.astype(np.float32) * sa.astype(np.float32)[:, None]) * sw.astype(np.float32)[None, :]
            return y if b is None else y + b.astype(np.float32)[None, :]
        assert np.array_equal(H.host(Y0), deq32(ref0, s_a0, s_w0, None)), "outputs differ (problem 0)"
        assert np.array_equal(H.host(Y1), deq32(ref1, s_a1, s_w1, bias1)), "outputs differ (problem 1)"
    else:
        H.assert_output_close(H.host(Y0), osg.dequant(ref0, s_a0, s_w0, None), out)
        H.assert_output_close(H.host(Y1), osg.dequant(ref1, s_a1, s_w1, bias1), out)
    Z0, Z1 = torch.empty_like(Y0), torch.empty_like(Y1)
    abi.w4a4_gemm(None, sa0, None, sw0, Z0, Xe=Xe0, We=We0)
    abi.w4a4_gemm(None, sa1, None, sw1, Z1, bias=b1, Xe=Xe1, We=We1)
    abi.check_status()
    assert torch.equal(Z0, Y0) and torch.equal(Z1, Y1), "grouped launch differs from single launches"


@pytest.mark.parametrize("M,N,K,dt", [(1, 32, 64, "f16"), (129, 288, 640, "f16"), (300, 512, 1024, "bf16"), (4608, 1024, 128, "bf16"),
                                      (1024, 4096, 4096, "f16"), (77, 768, 4096, "bf16")])
def test_fp16_gemm_ref(abi, M, N, K, dt):
    """The 16-bit baseline GEMM against the exact product: float64 sums of
    the 16-bit inputs; bound = one rounding to the element type plus float32
    accumulation error (2^-22 K^(1/2) of the sum of |a b| per output)."""
    rng = np.random.default_rng(M + N + K)
    A = rng.standard_normal((M, K)).astype(np.float32)
    B = rng.standard_normal((N, K)).astype(np.float32)
    if dt == "f16":
        A, B = A.astype(np.float16).astype(np.float32), B.astype(np.float16).astype(np.float32)
    else:
        A, B = inputs.round_to_bf16(A), inputs.round_to_bf16(B)
    C = torch.empty(M, N, dtype=H.torch_dtype(dt), device="cuda")
    abi.fp16_gemm_ref(H.dev(A, H.torch_dtype(dt)), H.dev(B, H.torch_dtype(dt)), C)
    abi.check_status()
    ref = A.astype(np.float64) @ B.astype(np.float64).T
    mag = np.abs(A).astype(np.float64) @ np.abs(B).astype(np.float64).T
    got = H.host(C).astype(np.float64)
    tol = H.half_spacing(ref, dt) + 2.0 ** -22 * np.sqrt(K) * mag
    if dt == "f16":
        tol = np.maximum(tol, 2.0 ** -11 * np.abs(ref)) + 2.0 ** -22 * np.sqrt(K) * mag
    assert np.all(np.abs(got - ref) <= tol), f"max excess {np.max(np.abs(got - ref) - tol)}"


@pytest.mark.parametrize("path", ["tma", "e4m3", "packed"])
@pytest.mark.parametrize("K", [18944, 65536])
def test_w4a4_gemm_adversarial_exactness(abi, K, path):
    """Integer exactness of the float32 tensor-core accumulation: all codes
    +-7 (largest accumulators), alternating signs, and a large running sum
    followed by increments of exactly 1 per 32-element MMA step (a truncating
    accumulator would drop them)."""
    L, N = 128, 256
    half = K // 2
    qa = np.zeros((L, K), np.int32)
    qw = np.zeros((N, K), np.int32)
    qa[0] = 7
    qw[0] = 7
    qw[1] = -7
    qa[1] = np.where(np.arange(K) % 2 == 0, 7, -7)
    qw[2] = np.where(np.arange(K) % 3 == 0, 7, -6)
    ramp_a = np.zeros(K, np.int32)
    ramp_a[:half] = 7
    ramp_a[half::32] = 1
    qa[2] = ramp_a
    qw[3] = ramp_a
    qw[4] = -ramp_a
    rng = np.random.default_rng(K)
    qa[3:] = rng.integers(-7, 8, (L - 3, K))
    qw[5:] = rng.integers(-7, 8, (N - 5, K))
    s_a = np.ones(L, np.float32)
    s_w = np.ones(N, np.float32)
    _, acc = run_gemm(abi, qa, qw, s_a, s_w, "f32", path=path)
    ref = osg.int_gemm(qa, qw)
    assert ref[0, 0] == 49 * K and ref[2, 3] == 49 * half + half // 32
    assert np.array_equal(acc, ref)


@pytest.mark.parametrize("g,L,C,zin,zout", [(4, 33, 64, "f16", "f32"), (8, 100, 256, "f16", "f16"),
                                            (16, 1025, 512, "bf16", "f32"), (32, 7, 96, "f32", "f32"),
                                            (64, 256, 512, "f16", "f32"), (128, 130, 4096, "f16", "f32"),
                                            (128, 64, 4096, "bf16", "bf16"),
                                            # more jobs than one wave: the streaming kernel with prepared
                                            # halves (runs crossing block boundaries, a ragged last tile)
                                            (128, 1407, 4096, "f16", "f16"), (64, 1201, 2048, "bf16", "f32"),
                                            (128, 8192, 3584, "bf16", "bf16")])
def test_tac_apply(abi, g, L, C, zin, zout):
    rng = np.random.default_rng(g * 1000 + L)
    Z = rng.standard_normal((L, C)).astype(np.float32)
    Z = Z.astype(np.float16).astype(np.float32) if zin == "f16" else (inputs.round_to_bf16(Z) if zin == "bf16" else Z)
    tp = inputs.make_tac(rng, C, g, noise=0.05)
    out = torch.empty(L, C, dtype=H.torch_dtype(zout), device="cuda")
    Zd, Md = H.dev(Z, H.torch_dtype(zin)), H.dev(tp.M)
    abi.tac_apply(Zd, Md, H.dev(tp.d), g, out)
    abi.check_status()
    ref = otac.tac_apply(Z, tp.M, tp.d, g)
    H.assert_tac_close(H.host(out), ref, zout)
    if zin != "f32" and g in (64, 128):
        # the prepared matrices (tac_prepare) give the same shared image, hence the same bits
        Mp = torch.empty(abi.tac_prepared_bytes(C, g), dtype=torch.uint8, device="cuda")
        abi.tac_prepare(Md, g, H.torch_dtype(zin), Mp)
        out2 = torch.empty_like(out)
        abi.tac_apply(Zd, Md, H.dev(tp.d), g, out2, Mp=Mp)
        abi.check_status()
        assert torch.equal(out2, out), "prepared TAC differs"


def _oracle_linear_from_codes(qa, s_a, qw, s_w, bias):
    acc = osg.int_gemm(qa, qw)
    return osg.dequant(acc, s_a, s_w, bias), acc


def run_linear_case(abi, case, out_dtype=None, check_rows=None, weights="e4m3"):
    """sgat_prepare_weight + sgat_linear on the GPU against the oracle's
    literal split / quantise / GEMM / scatter. With TAC, the TAC output is
    compared within tolerance and the rest of the chain is teacher-forced on
    the GPU's TAC output (left in the workspace in the input's type)."""
    xf = case.xf
    dt = H.torch_dtype(case.dtype)
    out_dtype = out_dtype or case.dtype
    L, K, N = case.L, case.K, case.N
    W = H.dev(case.W, dt)
    Wq = torch.empty(N, K // 2, dtype=torch.uint8, device="cuda")
    s_w = torch.empty(N, dtype=torch.float32, device="cuda")
    abi.sgat_prepare_weight(W, H.dev(xf.inv_a_w), xf.hb, Wq, s_w)
    We = unpacked_weight(abi, Wq) if weights == "e4m3" else None
    with_tac = case.tac is not None
    ws = torch.empty(abi.sgat_linear_workspace_size(L, K, with_tac), dtype=torch.uint8, device="cuda")
    Y = torch.empty(L, N, dtype=H.torch_dtype(out_dtype), device="cuda")
    kw = {}
    if with_tac:
        kw = dict(tac_M=H.dev(case.tac.M), tac_d=H.dev(case.tac.d), tac_g=case.tac.g)
        if weights == "e4m3" and case.dtype != "f32" and case.tac.g in (64, 128):
            # the main path also takes the prepared TAC matrices
            kw["tac_Mp"] = torch.empty(abi.tac_prepared_bytes(K, case.tac.g), dtype=torch.uint8, device="cuda")
            abi.tac_prepare(kw["tac_M"], case.tac.g, dt, kw["tac_Mp"])
    bias = H.dev(case.bias) if case.bias is not None else None
    abi.sgat_linear(H.dev(case.X, dt), H.dev(case.mask), H.dev(xf.a_m), H.dev(xf.a_u), xf.hb, xf.d_sh,
                    xf.d_m, xf.d_u, Wq, s_w, Y, ws, bias=bias, We=We, **kw)
    abi.check_status()
    qw, sw = osg.prepare_weight(case.W, xf.inv_a_w, xf.hb, 4)
    assert np.array_equal(H.unpack(Wq), qw) and np.array_equal(s_w.cpu().numpy(), sw)
    Xq_g, s_a_g, Xe_g, zt = H.workspace_views(ws, L, K, with_tac, dt)
    rows = np.arange(L) if check_rows is None else np.asarray(check_rows)
    X_in = case.X
    if with_tac:
        z_gpu = H.host(zt)
        ref_tac = otac.tac_apply(case.X[rows], case.tac.M, case.tac.d, case.tac.g)
        H.assert_tac_close(z_gpu[rows], ref_tac, case.dtype)
        X_in = z_gpu                      # teacher forcing on the GPU's TAC output
    Y_ref, codes, s_a, acc = osg.sgat_linear(X_in[rows], case.mask[rows], xf.a_m, xf.a_u, xf.hb, xf.d_sh,
                                             xf.d_m, xf.d_u, qw, sw, case.bias, 4)
    assert np.array_equal(H.codes_from_e4m3(Xe_g)[rows], codes), "activation codes differ"
    assert np.array_equal(Xe_g.cpu().numpy()[rows], H.e4m3_bytes(codes)), "E4M3 codes differ"
    assert np.array_equal(s_a_g.cpu().numpy()[rows], s_a), "activation scales differ"
    H.assert_output_close(H.host(Y)[rows], Y_ref, out_dtype)
    return Y


@pytest.mark.parametrize("weights", ["e4m3", "packed"])
@pytest.mark.parametrize("gates", [True, False])
def test_single_linear_full(abi, gates, weights):
    """Single SGAT linear, 256 x 512 -> 512, with and without gates, with
    and without TAC (block 64)."""
    case = inputs.single_linear(0, gates_on=gates)
    run_linear_case(abi, case, weights=weights)
    case.tac = None
    run_linear_case(abi, case, weights=weights)


@pytest.mark.parametrize("weights", ["e4m3", "packed"])
def test_llada_attention_full(abi, weights):
    """LLaDA-8B attention projections at one step: QKV 1024 x 4096 -> 12288
    and O 4096 -> 4096 with TAC (block 128), full size, every row."""
    qkv, o = inputs.llada_attention(0)
    run_linear_case(abi, qkv, weights=weights)
    run_linear_case(abi, o, weights=weights)


def _sample_rows(rng, L, n, mask):
    """Sorted sample of n rows with both states and both ends of the batch."""
    rows = set(rng.choice(L, n - 4, replace=False).tolist()) | {0, L - 1}
    rows |= {int(np.argmax(mask)), int(np.argmin(mask))}
    return np.array(sorted(rows))


@pytest.mark.parametrize("ratio", [0.1, 0.5, 0.9])
def test_llada_mlp(abi, ratio):
    """LLaDA-8B MLP at one step: gate+up 4096 -> 24576 with SGAT, SwiGLU
    (test glue on the GPU, in float32, rounded to float16), down 12288 ->
    4096 with SGAT on its own input (hb = 4096, three 4096-feature rounds
    per row). The mask is semi-autoregressive: the last round(32 ratio)
    blocks of 32 tokens are masked. Weight codes are compared for every
    channel, activations on 256 sampled tokens; the down projection is
    teacher-forced on the GPU's SwiGLU output."""
    gu, W_down, mask = inputs.llada_mlp(0, ratio)
    rng = np.random.default_rng(int(ratio * 10))
    rows = _sample_rows(rng, gu.L, 256, mask)
    Y = run_linear_case(abi, gu, check_rows=rows)
    F = gu.N // 2
    h = (torch.nn.functional.silu(Y[:, :F].float()) * Y[:, F:].float()).half()
    hx = h.float().cpu().numpy()
    down = inputs.LinearCase(f"llada_down_1024x12288x4096_r{ratio}", hx, "f16", mask, W_down,
                             inputs.make_sgat(hx, mask))
    assert down.xf.hb == 4096
    run_linear_case(abi, down, check_rows=rows)


def test_dream_block_linears(abi):
    """Dream-7B (Qwen2.5-7B shape) block linears on 4 x 2048 tokens in
    bfloat16: QKV with bias, O with TAC (block 128), gate+up 3584 -> 37888,
    down 18944 -> 3584 (hb = 512). Full-size launches; weight codes compared
    for every channel, activations and outputs on 256 sampled tokens."""
    cases = inputs.dream_block_linears(0)
    rng = np.random.default_rng(7)
    rows = _sample_rows(rng, cases[0].L, 256, cases[0].mask)
    for case in cases:
        run_linear_case(abi, case, check_rows=rows)


@pytest.mark.parametrize("L,K,F,dtype,bias", [(300, 512, 256, "f16", False), (77, 1024, 512, "bf16", True),
                                            (1024, 4096, 12288, "f16", False)])
def test_sgat_linear_swiglu(abi, L, K, F, dtype, bias):
    """Gate and up projections of a SwiGLU MLP with silu(gate) * up in the
    GEMM epilogue: the weight rows interleaved by swiglu_row_order, the
    output [L][F] against silu and the product taken in float64 from the
    oracle's dequantised gate and up outputs (the same float32 values the
    epilogue starts from). The last shape is the LLaDA-8B gate+up
    projection."""
    case = inputs.random_linear(L * 5 + K + F, L, K, 2 * F, dtype=dtype, bias=bias)
    xf = case.xf
    dt = H.torch_dtype(dtype)
    perm = abi.swiglu_row_order(F).numpy()
    Wp = case.W[perm]
    bp = case.bias[perm] if bias else None
    Wq = torch.empty(2 * F, K // 2, dtype=torch.uint8, device="cuda")
    s_w = torch.empty(2 * F, dtype=torch.float32, device="cuda")
    abi.sgat_prepare_weight(H.dev(Wp, dt), H.dev(xf.inv_a_w), xf.hb, Wq, s_w)
    We = unpacked_weight(abi, Wq)
    ws = torch.empty(abi.sgat_linear_workspace_size(L, K, False), dtype=torch.uint8, device="cuda")
    Hout = torch.full((L, F), float("nan"), dtype=dt, device="cuda")
    abi.sgat_linear_swiglu(H.dev(case.X, dt), H.dev(case.mask), H.dev(xf.a_m), H.dev(xf.a_u), xf.hb, xf.d_sh,
                           xf.d_m, xf.d_u, Wq, s_w, Hout, ws, bias=None if bp is None else H.dev(bp), We=We)
    abi.check_status()
    qw, sw = osg.prepare_weight(Wp, xf.inv_a_w, xf.hb, 4)
    Y_ref = osg.sgat_linear(case.X, case.mask, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, qw, sw, bp, 4)[0]
    Yr = Y_ref.reshape(L, F // 16, 2, 16)
    gate, up = Yr[:, :, 0, :].reshape(L, F), Yr[:, :, 1, :].reshape(L, F)
    h_ref = gate / (1.0 + np.exp(-gate)) * up
    H.assert_output_close(H.host(Hout), h_ref, dtype, what="silu(gate) * up")


@pytest.mark.parametrize("L,K,N,dtype,tac_g,bias", [(1, 128, 32, "f16", None, False),
                                                    (77, 512, 320, "bf16", 16, True),
                                                    (129, 1024, 256, "f16", 128, False),
                                                    (513, 3584, 512, "bf16", 128, True)])
@pytest.mark.parametrize("weights", ["e4m3", "packed"])
def test_sgat_linear_ragged(abi, L, K, N, dtype, tac_g, bias, weights):
    case = inputs.random_linear(L * 3 + K, L, K, N, dtype=dtype, tac_g=tac_g, bias=bias)
    run_linear_case(abi, case, weights=weights)


def test_empty_batch(abi):
    """L = 0 is a valid no-op for every entry point."""
    K, N = 512, 256
    X = torch.empty(0, K, dtype=torch.float16, device="cuda")
    Xq = torch.empty(0, K // 2, dtype=torch.uint8, device="cuda")
    s = torch.empty(0, dtype=torch.float32, device="cuda")
    abi.sgat_quantize_act(X, None, None, None, 512, K, 0, 0, Xq, s)
    Wq = torch.zeros(N, K // 2, dtype=torch.uint8, device="cuda")
    sw = torch.ones(N, dtype=torch.float32, device="cuda")
    Y = torch.empty(0, N, dtype=torch.float16, device="cuda")
    abi.w4a4_gemm(Xq, s, Wq, sw, Y)
    Xe0 = torch.empty(0, K, dtype=torch.uint8, device="cuda")
    abi.w4a4_gemm(None, s, Wq, sw, Y, Xe=Xe0)
    abi.w4a4_gemm(None, s, None, sw, Y, Xe=Xe0, We=unpacked_weight(abi, Wq))
    abi.w4_unpack_e4m3(torch.empty(0, K // 2, dtype=torch.uint8, device="cuda"),
                       torch.empty(0, K, dtype=torch.uint8, device="cuda"))
    abi.check_status()


@pytest.mark.parametrize("L,K,g,dtype,prepared", [(300, 1024, 64, "f16", True), (129, 4096, 128, "bf16", False),
                                                   (77, 512, 16, "f32", False)])
def test_quantize_act_tac_option(abi, L, K, g, dtype, prepared):
    """sgat_quantize_act with its tac option (Sec. 3.3: TAC on the attention
    output before the output projection's quantiser): the compensated rows in
    the scratch buffer within the TAC tolerance of the oracle's TAC, and the
    codes, scales and E4M3 bytes bit-exact with the oracle's quantiser on
    those rows (teacher-forced)."""
    case = inputs.random_linear(L * 3 + g, L, K, 128, dtype=dtype, tac_g=g)
    xf, tp = case.xf, case.tac
    dt = H.torch_dtype(dtype)
    X = H.dev(case.X, dt)
    Md = H.dev(tp.M)
    Mp = None
    if prepared:
        Mp = torch.empty(abi.tac_prepared_bytes(K, g), dtype=torch.uint8, device="cuda")
        abi.tac_prepare(Md, g, dt, Mp)
    scratch = torch.empty(L, K, dtype=dt, device="cuda")
    Xq = torch.empty(L, K // 2, dtype=torch.uint8, device="cuda")
    Xe = torch.empty(L, K, dtype=torch.uint8, device="cuda")
    s_a = torch.empty(L, dtype=torch.float32, device="cuda")
    abi.sgat_quantize_act(X, H.dev(case.mask), H.dev(xf.a_m), H.dev(xf.a_u), xf.hb, xf.d_sh, xf.d_m, xf.d_u, Xq, s_a,
                          Xe=Xe, tac_M=Md, tac_d=H.dev(tp.d), tac_g=g, tac_Mp=Mp, tac_scratch=scratch)
    abi.check_status()
    z = H.host(scratch)
    H.assert_tac_close(z, otac.tac_apply(case.X, tp.M, tp.d, g), dtype)
    codes, s = osg.sgat_quantize_act(z, case.mask, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, 4)
    assert np.array_equal(H.unpack(Xq), codes)
    assert np.array_equal(H.host(s_a), s)
    assert np.array_equal(H.host(Xe), H.e4m3_bytes(codes))


@pytest.mark.parametrize("L,N,K,g,dtype", [(256, 512, 512, 128, "f16"), (100, 384, 1024, 32, "bf16")])
def test_gemm_out_tac_option(abi, L, N, K, g, dtype):
    """w4a4_gemm with its out_tac option: the dequantised output in the
    scratch buffer within the output tolerance of the oracle, Y within the
    TAC tolerance of the oracle's TAC of that scratch output
    (teacher-forced), and the integer accumulators exact."""
    qa, qw, s_a, s_w = H.gemm_codes(L + N + K, L, N, K)
    rng = np.random.default_rng(g + L)
    tp = inputs.make_tac(rng, N, g, noise=0.05)
    dt = H.torch_dtype(dtype)
    Xe = H.dev(H.e4m3_bytes(qa))
    We = H.dev(H.e4m3_bytes(qw))
    Wq = H.dev(osg.pack_int4(qw))
    Y = torch.empty(L, N, dtype=dt, device="cuda")
    scratch = torch.empty(L, N, dtype=dt, device="cuda")
    acc = torch.empty(L, N, dtype=torch.int32, device="cuda")
    abi.w4a4_gemm(None, H.dev(s_a), Wq, H.dev(s_w), Y, acc_dbg=acc, Xe=Xe, We=We, tac_M=H.dev(tp.M),
                  tac_d=H.dev(tp.d), tac_g=g, tac_scratch=scratch)
    abi.check_status()
    ref_acc = osg.int_gemm(qa, qw)
    assert np.array_equal(H.host(acc), ref_acc)
    pre = H.host(scratch)
    H.assert_output_close(pre, osg.dequant(ref_acc, s_a, s_w, None), dtype, what="pre-TAC output")
    H.assert_tac_close(H.host(Y), otac.tac_apply(pre, tp.M, tp.d, g), dtype)


@pytest.mark.parametrize("L,N,K,out", [(1, 8, 128, "f32"), (200, 136, 512, "f16"), (129, 300, 1024, "bf16"),
                                       (1024, 4096, 4096, "f16")])
def test_gemm_mma_sync(abi, L, N, K, out):
    """The W4A4 GEMM on the warp-level int4 MMA (mma.sync m16n8k64 s4):
    int32 accumulators bit-exact with the oracle's integer product (ragged
    tiles, all-(-7) and all-(+7) rows for the extreme sums), outputs within
    the output tolerance, and the same outputs as w4a4_gemm's FP8-kind path
    bit for bit (the same float32 epilogue on the same exact sums)."""
    qa, qw, s_a, s_w = H.gemm_codes(L * 7 + N + K, L, N, K)
    qa[0] = -7
    qw[0] = -7
    if L > 1:
        qa[1] = 7
    Xq, Wq = H.dev(osg.pack_int4(qa)), H.dev(osg.pack_int4(qw))
    dt = H.torch_dtype(out)
    Y = torch.empty(L, N, dtype=dt, device="cuda")
    acc = torch.empty(L, N, dtype=torch.int32, device="cuda")
    abi.w4a4_gemm_mma_sync(Xq, H.dev(s_a), Wq, H.dev(s_w), Y, acc_dbg=acc)
    abi.check_status()
    ref = osg.int_gemm(qa, qw)
    assert np.array_equal(acc.cpu().numpy(), ref)
    assert ref[0, 0] == 49 * K
    H.assert_output_close(H.host(Y), osg.dequant(ref, s_a, s_w, None), out)
    if N % 32 == 0:
        Y2 = torch.empty_like(Y)
        abi.w4a4_gemm(Xq, H.dev(s_a), Wq, H.dev(s_w), Y2)
        abi.check_status()
        assert torch.equal(Y, Y2)
