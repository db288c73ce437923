"""Host-side checks of libstarq.so that need no GPU.

The library builds for sm_103a, loads, exports every function declared in
include/*.h, and rejects bad arguments with the documented error code before
any CUDA call (only validation paths run here: no compute call is made).
"""

import ctypes
import os
import re

import pytest

from tests.conftest import ROOT


def declared_functions():
    names = []
    inc = os.path.join(ROOT, "include")
    for fn in sorted(os.listdir(inc)):
        if not fn.endswith(".h"):
            continue
        src = open(os.path.join(inc, fn)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w \*]*?\b([A-Za-z_]\w*)\s*\(", src, flags=re.M):
            if not src[m.start():].startswith(("typedef", "enum", "struct", "#")):
                names.append(m.group(1))
    return sorted(set(names))


@pytest.fixture(scope="module")
def lib():
    from paper_2606_04945_gb300 import build
    build.build()
    from paper_2606_04945_gb300 import abi
    return abi


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert "sgat_linear" in names and "w4a4_gemm" in names and len(names) >= 9
    for n in names:
        assert hasattr(lib.lib, n), n
    assert set(lib.EXPORTED) <= set(names)


def test_version_and_last_error(lib):
    assert lib.lib.starq_version() >= 100
    assert isinstance(lib.lib.starq_last_error(), bytes)


P = ctypes.c_void_p(4096)  # a non-null, 16-byte-aligned stand-in; never dereferenced


@pytest.mark.parametrize("args,code", [
    ((None, 0, 4, 512, None, None, None, 512, 512, 0, 0, None, 4, P, P, None, None, None), -1),   # NULL X
    ((P, 9, 4, 512, None, None, None, 512, 512, 0, 0, None, 4, P, P, None, None, None), -1),      # dtype
    ((P, 0, 4, 512, None, None, None, 512, 512, 0, 0, None, 6, P, P, None, None, None), -4),      # bits (4 or 8)
    ((P, 0, 4, 100, None, None, None, 4, 100, 0, 0, None, 4, P, P, None, None, None), -2),        # K % 16
    ((P, 0, 4, 512, None, None, None, 384, 512, 0, 0, None, 4, P, P, None, None, None), -2),      # hb not pow2
    ((P, 0, 4, 512, None, None, None, 8192, 512, 0, 0, None, 4, P, P, None, None, None), -2),     # hb > K
    ((P, 0, 4, 512, None, None, None, 512, 500, 6, 0, None, 4, P, P, None, None, None), -2),      # gate sum
    ((P, 0, -1, 512, None, None, None, 512, 512, 0, 0, None, 4, P, P, None, None, None), -2),     # L < 0
    ((ctypes.c_void_p(4100), 0, 4, 512, None, None, None, 512, 512, 0, 0, None, 4, P, P, None, None, None), -3),
])
def test_quantize_act_validation(lib, args, code):
    assert lib.lib.sgat_quantize_act(*args) == code
    assert lib.lib.starq_last_error()


@pytest.mark.parametrize("L,N,K,code", [(4, 96, 512, -2), (4, 256, 200, -2), (4, 256, 131072, -2),
                                        (-1, 256, 512, -2), (4, 256, 512, -1)])
def test_w8a8_gemm_validation(lib, L, N, K, code):
    """8-bit GEMM: N % 128, K % 128, K <= 65536, L >= 0; NULL Xe with L > 0."""
    Xe = None if code == -1 else P
    assert lib.lib.w8a8_gemm(Xe, P, P, P, None, L, N, K, P, 0, None, None) == code
    assert lib.lib.starq_last_error()


def test_w8_codes_validation(lib):
    assert lib.lib.w8_codes_f16(P, 4, 200, P, None) == -2           # K % 128
    assert lib.lib.w8_codes_f16(ctypes.c_void_p(4100), 4, 256, P, None) == -3
    assert lib.lib.w8_codes_f16(P, 0, 256, P, None) == 0            # nothing to do


def test_linear_workspace_by_bits(lib):
    """8-bit codes take a byte each and their fp16 operand form two; 4-bit
    codes half a byte and one."""
    L, K = 1000, 4096
    a256 = lambda x: (x + 255) // 256 * 256
    assert lib.lib.sgat_linear_workspace_size_bits(L, K, 0, 4) == lib.lib.sgat_linear_workspace_size(L, K, 0)
    assert lib.lib.sgat_linear_workspace_size_bits(L, K, 0, 8) == a256(L * K) + a256(4 * L) + a256(2 * L * K)
    assert lib.lib.sgat_linear_workspace_size_bits(L, K, 1, 8) == (a256(L * K) + a256(4 * L) + a256(2 * L * K)
                                                                   + a256(4 * L * K))
    assert lib.lib.sgat_linear_workspace_size_bits(L, K, 0, 6) == 0


def W4(lib, *args):
    """w4a4_gemm with out_tac = NULL (the argument before acc_dbg)."""
    return lib.lib.w4a4_gemm(*args[:12], None, *args[12:])


@pytest.mark.parametrize("L,N,K,code", [(4, 100, 512, -2), (4, 256, 200, -2), (4, 256, 131072, -2),
                                        (-1, 256, 512, -2)])
def test_gemm_validation(lib, L, N, K, code):
    assert W4(lib, P, None, P, P, None, P, None, L, N, K, P, 0, None, None) == code


def test_gemm_null_and_alignment(lib):
    assert W4(lib, None, None, P, P, None, P, None, 4, 256, 512, P, 0, None, None) == -1
    assert W4(lib, P, None, P, None, None, P, None, 4, 256, 512, P, 0, None, None) == -1
    # E4M3 weights need E4M3 activations when there are no packed weights
    assert W4(lib, P, None, P, None, P, P, None, 4, 256, 512, P, 0, None, None) == -1
    assert W4(lib, ctypes.c_void_p(4104), None, P, P, None, P, None, 4, 256, 512, P, 0, None, None) == -3
    assert W4(lib, None, ctypes.c_void_p(4104), P, P, None, P, None, 4, 256, 512, P, 0, None, None) == -3
    assert W4(lib, None, P, P, None, ctypes.c_void_p(4104), P, None, 4, 256, 512, P, 0, None, None) == -3
    assert W4(lib, P, None, P, P, None, P, None, 4, 256, 512, P, 7, None, None) == -1


def Q2(lib, X0=P, Xq1=P, d_m=0, hb=512, bits=4, L=4, K=512, dt=0, none=None):
    """sgat_quantize_act_grouped with valid placeholder problems except
    where overridden (validation returns before any device access)."""
    io = lambda X, Xq: lib.StarqQuantIo(X, None, None, None, K, d_m, 0, Xq, P, None)
    p0, p1 = io(X0, P), io(P, Xq1)
    args = [ctypes.byref(p0), ctypes.byref(p1)]
    if none is not None:
        args[none] = None
    return lib.lib.sgat_quantize_act_grouped(*args, dt, L, K, hb, bits, None)


def test_quantize_grouped_validation(lib):
    assert Q2(lib, none=0) == -1
    assert Q2(lib, none=1) == -1
    assert Q2(lib, Xq1=None) == -1
    assert Q2(lib, dt=7) == -1
    assert Q2(lib, bits=6) == -4
    assert Q2(lib, hb=3) == -2
    assert Q2(lib, d_m=5) == -2                       # d_sh + d_m + d_u != K
    assert Q2(lib, L=-1) == -2
    assert Q2(lib, X0=ctypes.c_void_p(4104)) == -3
    assert Q2(lib, L=0, X0=None, Xq1=None) == 0


def G2(lib, Xe0=P, We0=P, N0=256, Y0=P, Xe1=P, We1=P, N1=128, L=4, K=512, dt=0, acc0=None, flags=0):
    """w4a4_gemm_grouped with valid placeholders except where overridden
    (validation returns before any device access)."""
    return lib.lib.w4a4_gemm_grouped(Xe0, P, We0, P, None, N0, Y0, Xe1, P, We1, P, None, N1, P, L, K, dt, acc0,
                                     None, flags, None)


@pytest.mark.parametrize("N0,N1,K,L,code", [(100, 256, 512, 4, -2), (256, 31, 512, 4, -2), (256, 256, 200, 4, -2),
                                            (256, 256, 131072, 4, -2), (256, 256, 512, -1, -2)])
def test_gemm_grouped_validation(lib, N0, N1, K, L, code):
    assert G2(lib, N0=N0, N1=N1, K=K, L=L) == code


def test_gemm_grouped_null_and_alignment(lib):
    assert G2(lib, We0=None) == -1
    assert G2(lib, We1=None) == -1
    assert G2(lib, Xe1=None) == -1
    assert G2(lib, Xe0=ctypes.c_void_p(4104)) == -3
    assert G2(lib, We1=ctypes.c_void_p(4104)) == -3
    assert G2(lib, Y0=ctypes.c_void_p(4104)) == -3
    assert G2(lib, acc0=ctypes.c_void_p(4100)) == -3
    assert G2(lib, dt=7) == -1
    assert G2(lib, flags=2) == -1
    assert G2(lib, L=0, Xe0=None, Xe1=None) == 0
    assert G2(lib, L=0, Xe0=None, Xe1=None, flags=1) == 0


@pytest.mark.parametrize("N,K,code", [(-1, 512, -2), (4, 48, -2), (4, 16, -2)])
def test_unpack_validation(lib, N, K, code):
    assert lib.lib.w4_unpack_e4m3(P, N, K, P, None) == code


def test_unpack_null_and_alignment(lib):
    assert lib.lib.w4_unpack_e4m3(None, 4, 512, P, None) == -1
    assert lib.lib.w4_unpack_e4m3(P, 4, 512, ctypes.c_void_p(4100), None) == -3
    assert lib.lib.w4_unpack_e4m3(None, 0, 512, None, None) == 0


@pytest.mark.parametrize("M,N,K,dt,code", [(4, 100, 512, 0, -2), (4, 256, 96, 0, -2), (-1, 256, 512, 0, -2),
                                            (4, 256, 512, 2, -1), (0, 256, 512, 0, 0)])
def test_fp16_gemm_validation(lib, M, N, K, dt, code):
    assert lib.lib.fp16_gemm_ref(P, P, dt, M, N, K, P, None) == code


def test_fp16_gemm_alignment(lib):
    assert lib.lib.fp16_gemm_ref(ctypes.c_void_p(4098), P, 0, 4, 256, 512, P, None) == -3
    assert lib.lib.fp16_gemm_ref(None, P, 0, 4, 256, 512, P, None) == -1


@pytest.mark.parametrize("g,C,code", [(12, 96, -2), (16, 100, -2), (256, 4096, -2)])
def test_tac_validation(lib, g, C, code):
    assert lib.lib.tac_apply(P, 0, 4, C, g, P, P, None, P, 0, None) == code


def test_tac_null_matrix(lib):
    assert lib.lib.tac_apply(P, 0, 4, 64, 16, None, P, None, P, 0, None) == -1


def test_tac_prepared_only_on_the_tensor_core_path(lib):
    assert lib.lib.tac_apply(P, 2, 4, 256, 128, P, P, P, P, 2, None) == -1      # float32 Z
    assert lib.lib.tac_apply(P, 0, 4, 256, 32, P, P, P, P, 2, None) == -1      # g = 32
    assert lib.lib.tac_apply(P, 0, 4, 256, 128, P, P, ctypes.c_void_p(4104), P, 2, None) == -3


@pytest.mark.parametrize("C,g,dt,code", [(256, 32, 0, -2), (200, 64, 0, -2), (256, 128, 2, -1), (0, 128, 1, 0)])
def test_tac_prepare_validation(lib, C, g, dt, code):
    assert lib.lib.tac_prepare(P, C, g, dt, P, None) == code


def test_tac_prepare_null_and_alignment(lib):
    assert lib.lib.tac_prepare(None, 256, 128, 0, P, None) == -1
    assert lib.lib.tac_prepare(P, 256, 128, 0, ctypes.c_void_p(4100), None) == -3


def test_linear_workspace_and_validation(lib):
    n = lib.sgat_linear_workspace_size(1024, 4096, False)
    assert n == 1024 * 2048 + 4096 + 1024 * 4096
    assert lib.sgat_linear_workspace_size(1024, 4096, True) == n + 1024 * 4096 * 4
    # workspace too small
    rc = lib.lib.sgat_linear(P, 0, 1024, 4096, None, None, None, 4096, 4096, 0, 0, None, None, 0, None,
                             P, None, P, None, 256, 4, P, 0, P, 16, None)
    assert rc == -2 and b"workspace" in lib.lib.starq_last_error()
    # TAC block that does not divide K
    rc = lib.lib.sgat_linear(P, 0, 16, 4096, None, None, None, 4096, 4096, 0, 0, P, None, 48, None,
                             P, None, P, None, 256, 4, P, 0, P, 1 << 30, None)
    assert rc == -2


def test_tac_calibrate_validation(lib):
    """Argument checks of tac_calibrate run before any CUDA call."""
    L = lib.lib
    ws = lib.tac_calibrate_workspace_size(4096, 128)
    assert ws == (4096 // 128) * (2 * 128 + 5 * 128 * 128) * 8
    assert lib.tac_calibrate_workspace_size(100, 16) == 0                          # C % g != 0
    good = dict(zf=P, zq=P, dt=0, N=64, C=256, g=16, rho=3e-4, eps=1e-8, eta=0.15, alpha=0.55, M=P, d=P,
                w=ctypes.c_void_p(4096), wb=lib.tac_calibrate_workspace_size(256, 16))

    def call(**kw):
        a = dict(good, **kw)
        return L.tac_calibrate(a["zf"], a["zq"], a["dt"], a["N"], a["C"], a["g"], a["rho"], a["eps"], a["eta"],
                               a["alpha"], a["M"], a["d"], a["w"], a["wb"], None)
    assert call(zf=None) == -1 and call(M=None) == -1 and call(w=None) == -1
    assert call(dt=5) == -1
    assert call(g=12) == -2 and call(g=256) == -2 and call(C=100) == -2 and call(N=0) == -2
    assert call(eps=0.0) == -1 and call(eta=1.5) == -1 and call(alpha=-0.1) == -1 and call(rho=-1.0) == -1
    assert call(wb=good["wb"] - 8) == -2
    assert call(zq=ctypes.c_void_p(4104)) == -3 and call(w=ctypes.c_void_p(4104)) == -3
    assert "tac_calibrate" in L.starq_last_error().decode()


def test_asym_validation(lib):
    """Asymmetric entry points: NULL zero points, the zero-point columns' K
    limits (K % 128, K <= 7680), alignment; the workspace layout."""
    L, K = 4, 512
    args = lambda z, k, xe, x=P: (x, 0, L, k, None, None, None, 1, k, 0, 0, P, P, z, xe, None)
    assert lib.lib.sgat_quantize_act_asym(*args(None, K, P)) == -1
    assert lib.lib.sgat_quantize_act_asym(*args(P, 528, P)) == -2          # Xe needs K % 128
    assert lib.lib.sgat_quantize_act_asym(*args(P, 7808, P)) == -2         # above 7680
    assert lib.lib.sgat_quantize_act_asym(*args(P, K, ctypes.c_void_p(4104))) == -3
    assert lib.lib.w4_zero_point_columns(P, 4, 7808, P, None) == -2
    assert lib.lib.w4_zero_point_columns(P, 4, 200, P, None) == -2
    assert lib.lib.w4_zero_point_columns(ctypes.c_void_p(4100), 4, 256, P, None) == -3
    assert lib.lib.w4_zero_point_columns(P, 0, 256, P, None) == 0
    a256 = lambda x: (x + 255) // 256 * 256
    assert lib.lib.sgat_linear_asym_workspace_size(1000, 4096) == (a256(1000 * 2048) + 2 * a256(4000)
                                                                   + a256(1000 * 4224))
    assert lib.lib.sgat_linear_asym(P, 0, L, 8192, None, None, None, 1, 8192, 0, 0, P, P, None, 64, P, 0, P,
                                    1 << 30, None) == -2


def test_dense_validation(lib):
    """Dense-basis entry points: NULL basis, K limits (K % 128, K <= 16384),
    a short workspace; the workspace sizes."""
    L, K = 4, 512
    q = lambda pt, k, wsb: lib.lib.sgat_quantize_act_dense(P, 0, L, k, None, None, None, pt, k, 0, 0, P, P, None, P,
                                                           wsb, None)
    assert q(None, K, 1 << 20) == -1
    assert q(P, 576, 1 << 20) == -2
    assert q(P, 16512, 1 << 30) == -2
    assert q(P, K, 100) == -2
    assert lib.lib.sgat_prepare_weight_dense(P, 0, 4, K, None, None, P, P, P, 1 << 20, None) == -1
    a256 = lambda x: (x + 255) // 256 * 256
    assert lib.lib.sgat_dense_workspace_size(100, 1024) == 2 * a256(100 * 1024 * 2)
    assert lib.lib.sgat_linear_dense_workspace_size(100, 1024) == (2 * a256(100 * 1024 * 2) + a256(100 * 512)
                                                                   + a256(400) + a256(100 * 1024))


def test_zero_point_decomposition_rule_covers_the_k_limit():
    """The weight-side zero-point columns hold sum_k q_w as 448s plus a
    greedy remainder of E4M3 numbers (each step takes the largest E4M3
    value not above what is left). For every |sum| <= 7 K at the API's
    limit K = 7680 this ends exactly within 128 columns, and every term is
    an E4M3 number. The rule is written here from the format's definition
    (3 mantissa bits: above 16, values 2^e (1 + m/8))."""
    def e4m3_floor(r):
        if r <= 16:
            return r
        e = r.bit_length() - 1
        step = 1 << (e - 3)
        return min(r // step * step, 448)

    def is_e4m3(v):
        if v <= 16:
            return True
        e = v.bit_length() - 1
        return v <= 448 and v % (1 << (e - 3)) == 0

    worst = 0
    for mag in range(0, 7 * 7680 + 1):
        n448, rem = divmod(mag, 448)
        terms = []
        while rem:
            t = e4m3_floor(rem)
            assert is_e4m3(t)
            terms.append(t)
            rem -= t
        assert len(terms) <= 5
        worst = max(worst, n448 + len(terms))
    assert worst <= 128


def test_validation_from_eight_threads(lib):
    """Eight host threads call validation-only paths at once. Each thread
    gets its own return code and its own last-error message (the message is
    per thread), and calls that pass validation reach the per-device caches
    (which on a machine without a GPU fail cleanly with STARQ_ERR_CUDA
    instead of racing)."""
    import threading
    import torch

    lib_ = lib.lib
    gpu = torch.cuda.is_available()
    errors = []
    barrier = threading.Barrier(8)

    def worker(t):
        try:
            barrier.wait()
            for it in range(200):
                K = 100 + 16 * t                     # K % 16 != 0 for every t: a shape error
                rc = lib_.sgat_quantize_act(P, 0, 4, K, None, None, None, 4, K, 0, 0, None, 4, P, P, None, None, None)
                msg = lib_.starq_last_error().decode()
                if rc != -2 or f"K={K}" not in msg:
                    errors.append((t, it, rc, msg))
                rc = lib_.w8a8_gemm(P, P, P, P, None, 4, 96 + 0 * t, 512, P, 0, None, None)
                if rc != -2:
                    errors.append((t, it, "w8a8", rc))
                if not gpu:
                    # valid arguments: the call reaches the device-side lookups and
                    # fails there without a device
                    rc = lib_.tac_prepare(P, 256, 64, 0, P, None)
                    if rc != lib.ERR_CUDA:
                        errors.append((t, it, "tac_prepare", rc))
        except Exception as e:  # pragma: no cover
            errors.append((t, repr(e)))

    threads = [threading.Thread(target=worker, args=(t,)) for t in range(8)]
    for th in threads:
        th.start()
    for th in threads:
        th.join()
    assert not errors, errors[:5]


@pytest.mark.parametrize("g,M,Mp,scratch,dtype,code", [
    (5, P, None, P, 0, -2),                          # block size
    (64, None, None, P, 0, -1),                      # no M
    (64, P, None, None, 0, -1),                      # no scratch buffer
    (64, P, None, ctypes.c_void_p(4104), 0, -3),     # scratch alignment
    (16, P, P, P, 0, -1),                            # prepared M only for g = 64 / 128
    (64, P, P, P, 2, -1),                            # prepared M only for 16-bit tensors
])
def test_tac_option_validation(lib, g, M, Mp, scratch, dtype, code):
    """The tac option of sgat_quantize_act (TAC on the input) and the out_tac
    option of w4a4_gemm (TAC on the output) are validated before any launch."""
    from paper_2606_04945_gb300.abi import StarqTac
    v = lambda p: None if p is None else p.value
    t = StarqTac(g, v(M), None, v(Mp), v(scratch))
    assert lib.lib.sgat_quantize_act(P, dtype, 4, 512, None, None, None, 512, 512, 0, 0, ctypes.byref(t), 4, P, P,
                                     None, None, None) == code
    assert lib.lib.starq_last_error()
    assert lib.lib.w4a4_gemm(P, None, P, P, None, P, None, 4, 256, 512, P, dtype, ctypes.byref(t), None,
                             None) == (code if g != 5 else -2)


def test_gemm_pair_limit(lib):
    """The pair cap is thread-local state: it returns the previous cap and
    rejects negative values without touching it."""
    prev = lib.set_gemm_pair_limit(48)
    try:
        assert lib.set_gemm_pair_limit(12) == 48
        with pytest.raises(lib.StarqError):
            lib.set_gemm_pair_limit(-1)
        assert lib.set_gemm_pair_limit(0) == 12
    finally:
        lib.set_gemm_pair_limit(prev)
