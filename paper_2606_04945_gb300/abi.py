"""Python binding of libstarq.so (include/starq.h): argument marshalling only.

Every function takes torch CUDA tensors, passes their device pointers and
sizes to the C ABI, and raises ``StarqError`` with the library's message on
a non-zero return. No step of the computation runs in Python: if the
library is missing or fails to load, importing this module raises.
"""

import ctypes
import os

import torch

from .build import LIB

F16, BF16, F32 = 0, 1, 2
OK, ERR_ARG, ERR_SHAPE, ERR_ALIGN, ERR_BITS, ERR_CUDA, ERR_TIMEOUT = 0, -1, -2, -3, -4, -5, -6

EXPORTED = (
    "starq_version", "starq_last_error", "starq_check_status",
    "sgat_quantize_act", "sgat_prepare_weight", "w4_unpack_e4m3", "w4a4_gemm", "fp16_gemm_ref", "tac_prepare", "tac_apply",
    "sgat_linear_workspace_size", "sgat_linear", "starq_last_gemm_tile",
    "tac_calibrate_workspace_size", "tac_calibrate", "sgat_linear_swiglu",
    "attention_pv_tac_workspace_size", "attention_pv_tac",
    "w8_codes_f16", "w8a8_gemm", "sgat_linear_workspace_size_bits",
    "sgat_quantize_act_asym", "w4_zero_point_columns", "sgat_linear_asym_workspace_size", "sgat_linear_asym",
    "sgat_dense_workspace_size", "sgat_quantize_act_dense", "sgat_prepare_weight_dense",
    "sgat_linear_dense_workspace_size", "sgat_linear_dense", "sgat_linear_noalloc",
    "starq_selftest_wait_timeout", "starq_probe_mma", "attention_pv_tac_gqa", "glue_add_rmsnorm", "glue_rope",
    "w4a4_gemm_mma_sync", "starq_set_gemm_pair_limit", "w4a4_gemm_grouped", "sgat_quantize_act_grouped",
)


class StarqQuantIo(ctypes.Structure):
    """starq_quant_io: one problem of sgat_quantize_act_grouped."""
    _fields_ = [("X", ctypes.c_void_p), ("mask", ctypes.c_void_p), ("a_m", ctypes.c_void_p),
                ("a_u", ctypes.c_void_p), ("d_sh", ctypes.c_int), ("d_m", ctypes.c_int), ("d_u", ctypes.c_int),
                ("Xq", ctypes.c_void_p), ("s_a", ctypes.c_void_p), ("Xe", ctypes.c_void_p),
                ("independent", ctypes.c_int)]


class StarqTac(ctypes.Structure):
    """starq_tac: TAC parameters of the tac option of sgat_quantize_act and
    w4a4_gemm."""
    _fields_ = [("g", ctypes.c_int), ("M", ctypes.c_void_p), ("d", ctypes.c_void_p), ("Mp", ctypes.c_void_p),
                ("scratch", ctypes.c_void_p)]


def _tac_struct(M, d, g, Mp, scratch):
    """A StarqTac for the given tensors, or None when M is None."""
    if M is None:
        return None
    _contig(M, d, Mp, scratch)
    ptr = lambda t: None if t is None else t.data_ptr()
    return StarqTac(int(g), ptr(M), ptr(d), ptr(Mp), ptr(scratch))


def _ref(struct):
    return None if struct is None else ctypes.byref(struct)


class StarqError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"starq error {code}: {msg}")
        self.code = code


def _load():
    if not os.path.exists(LIB):
        raise ImportError(
            f"{LIB} is missing: build it first (python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(LIB)
    vp, i, f_p, u8p = ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p
    lib.starq_version.restype = i
    lib.starq_last_error.restype = ctypes.c_char_p
    lib.starq_check_status.argtypes = [vp]
    lib.starq_selftest_wait_timeout.argtypes = [ctypes.c_uint, vp]
    lib.glue_add_rmsnorm.argtypes = [vp, vp, i, i, i, f_p, ctypes.c_float, vp, vp, vp]
    lib.glue_rope.argtypes = [vp, i, i, i, i, vp, ctypes.c_double, vp]
    lib.starq_probe_mma.argtypes = [i, i, vp, vp, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_double), vp]
    lib.sgat_quantize_act.argtypes = [vp, i, i, i, u8p, f_p, f_p, i, i, i, i, vp, i, u8p, f_p, u8p, f_p, vp]
    lib.sgat_prepare_weight.argtypes = [vp, i, i, i, f_p, i, i, u8p, f_p, vp]
    lib.w4_unpack_e4m3.argtypes = [u8p, i, i, u8p, vp]
    lib.w4a4_gemm.argtypes = [u8p, u8p, f_p, u8p, u8p, f_p, f_p, i, i, i, vp, i, vp, vp, vp]
    lib.w8_codes_f16.argtypes = [u8p, i, i, u8p, vp]
    lib.w4a4_gemm_mma_sync.argtypes = [u8p, f_p, u8p, f_p, f_p, i, i, i, vp, i, vp, vp]
    lib.sgat_quantize_act_grouped.argtypes = [vp, vp, i, i, i, i, i, vp]
    lib.w4a4_gemm_grouped.argtypes = [u8p, f_p, u8p, f_p, f_p, i, vp, u8p, f_p, u8p, f_p, f_p, i, vp, i, i, i, vp,
                                      vp, i, vp]
    lib.starq_set_gemm_pair_limit.argtypes = [i]
    lib.starq_set_gemm_pair_limit.restype = i
    lib.w8a8_gemm.argtypes = [u8p, f_p, u8p, f_p, f_p, i, i, i, vp, i, vp, vp]
    lib.sgat_linear_workspace_size_bits.argtypes = [i, i, i, i]
    lib.sgat_linear_workspace_size_bits.restype = ctypes.c_size_t
    lib.sgat_quantize_act_asym.argtypes = [vp, i, i, i, u8p, f_p, f_p, i, i, i, i, u8p, f_p, vp, u8p, vp]
    lib.w4_zero_point_columns.argtypes = [u8p, i, i, u8p, vp]
    lib.sgat_linear_asym_workspace_size.argtypes = [i, i]
    lib.sgat_linear_asym_workspace_size.restype = ctypes.c_size_t
    lib.sgat_linear_asym.argtypes = [vp, i, i, i, u8p, f_p, f_p, i, i, i, i, u8p, f_p, f_p, i, vp, i, vp,
                                     ctypes.c_size_t, vp]
    lib.sgat_dense_workspace_size.argtypes = [i, i]
    lib.sgat_dense_workspace_size.restype = ctypes.c_size_t
    lib.sgat_quantize_act_dense.argtypes = [vp, i, i, i, u8p, f_p, f_p, vp, i, i, i, u8p, f_p, u8p, vp,
                                            ctypes.c_size_t, vp]
    lib.sgat_prepare_weight_dense.argtypes = [vp, i, i, i, f_p, vp, u8p, f_p, vp, ctypes.c_size_t, vp]
    lib.sgat_linear_dense_workspace_size.argtypes = [i, i]
    lib.sgat_linear_dense_workspace_size.restype = ctypes.c_size_t
    lib.sgat_linear_dense.argtypes = [vp, i, i, i, u8p, f_p, f_p, vp, i, i, i, u8p, u8p, f_p, f_p, i, vp, i, vp,
                                      ctypes.c_size_t, vp]
    lib.tac_prepare.argtypes = [f_p, i, i, i, vp, vp]
    lib.starq_last_gemm_tile.restype = i
    dbl = ctypes.c_double
    lib.tac_calibrate_workspace_size.argtypes = [i, i]
    lib.tac_calibrate_workspace_size.restype = ctypes.c_size_t
    lib.tac_calibrate.argtypes = [vp, vp, i, i, i, i, dbl, dbl, dbl, dbl, f_p, f_p, vp, ctypes.c_size_t, vp]
    lib.tac_apply.argtypes = [vp, i, i, i, i, f_p, f_p, vp, vp, i, vp]
    lib.fp16_gemm_ref.argtypes = [vp, vp, i, i, i, i, vp, vp]
    lib.sgat_linear_workspace_size.argtypes = [i, i, i]
    lib.sgat_linear_workspace_size.restype = ctypes.c_size_t
    lib.sgat_linear.argtypes = [vp, i, i, i, u8p, f_p, f_p, i, i, i, i, f_p, f_p, i, vp,
                                u8p, u8p, f_p, f_p, i, i, vp, i, vp, ctypes.c_size_t, vp]
    lib.sgat_linear_swiglu.argtypes = lib.sgat_linear.argtypes
    lib.attention_pv_tac_workspace_size.argtypes = [i, i]
    lib.attention_pv_tac_workspace_size.restype = ctypes.c_size_t
    lib.attention_pv_tac.argtypes = [vp, vp, vp, i, i, i, vp, f_p, vp, vp, vp, vp, vp, ctypes.c_size_t, vp]
    lib.attention_pv_tac_gqa.argtypes = [vp, vp, vp, i, i, i, i, i, vp, f_p, vp, vp, vp, vp, vp, ctypes.c_size_t,
                                         vp]
    lib.sgat_linear_noalloc.argtypes = [vp, i, i, i, u8p, f_p, f_p, i, i, i, i, f_p, f_p, i, vp,
                                        u8p, u8p, f_p, f_p, i, i, vp, i, vp]
    return lib


lib = _load()


def _check(rc):
    if rc != 0:
        raise StarqError(rc, lib.starq_last_error().decode())


def dtype_code(t):
    return {torch.float16: F16, torch.bfloat16: BF16, torch.float32: F32}[t.dtype]


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _contig(*ts):
    for t in ts:
        if t is not None and not t.is_contiguous():
            raise ValueError("starq expects contiguous tensors")


def check_status(stream=None):
    """Synchronise and raise if a kernel gave up a bounded wait."""
    _check(lib.starq_check_status(_stream(stream)))


def selftest_wait_timeout(limit_us, stream=None):
    """Launch the bounded-wait self-test kernel (a wait on a barrier nobody
    arms, given up after limit_us); the next check_status raises
    StarqError(ERR_TIMEOUT)."""
    _check(lib.starq_selftest_wait_timeout(int(limit_us), _stream(stream)))


PROBE_KINDS = {0: "tcgen05 kind::f8f6f4 cta_group::1 M128 N256 K32 (E4M3)",
               1: "tcgen05 kind::f8f6f4 cta_group::2 M256 N256 K32 (E4M3, CTA pairs)",
               2: "tcgen05 kind::f16 cta_group::1 M128 N256 K16 (bf16)",
               3: "mma.sync m16n8k32 s8.s8.s32",
               4: "mma.sync m16n8k64 s4.s4.s32"}


def probe_mma(kind, iters, cycles, errors, stream=None):
    """Launch the tensor-core rate probe; cycles (int64 [4 * SMs]) and errors
    (int32 [1], zeroed) are device tensors. Returns (ctas, macs_per_cta)."""
    ctas = ctypes.c_int(0)
    macs = ctypes.c_double(0.0)
    _check(lib.starq_probe_mma(int(kind), int(iters), _p(cycles), _p(errors), ctypes.byref(ctas),
                               ctypes.byref(macs), _stream(stream)))
    return ctas.value, macs.value


def sgat_quantize_act(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, Xq, s_a, bits=4, Xe=None, v_dbg=None,
                      stream=None, tac_M=None, tac_d=None, tac_g=0, tac_Mp=None, tac_scratch=None):
    """With tac_M: TAC on X first (into tac_scratch [L][K], X's type), then
    the quantiser on the compensated rows."""
    _contig(X, mask, a_m, a_u, Xq, s_a, Xe, v_dbg)
    L, K = X.shape
    tac = _tac_struct(tac_M, tac_d, tac_g, tac_Mp, tac_scratch)
    _check(lib.sgat_quantize_act(_p(X), dtype_code(X), L, K, _p(mask), _p(a_m), _p(a_u), hb,
                                 d_sh, d_m, d_u, _ref(tac), bits, _p(Xq), _p(s_a), _p(Xe), _p(v_dbg),
                                 _stream(stream)))


def sgat_quantize_act_grouped(p0, p1, hb, bits=4, stream=None):
    """Two quantisations in one launch. p0, p1: dicts with X [L][K], mask,
    a_m, a_u, d_sh, d_m, d_u, Xq, s_a and optionally Xe (the meanings of
    sgat_quantize_act) and independent (see starq_quant_io); the two X share
    shape and dtype."""
    X0, X1 = p0["X"], p1["X"]
    if tuple(X0.shape) != tuple(X1.shape) or X0.dtype != X1.dtype:
        raise StarqError(-2, "sgat_quantize_act_grouped: the inputs need the same shape and dtype")
    ios = []
    for p in (p0, p1):
        _contig(p["X"], p.get("mask"), p.get("a_m"), p.get("a_u"), p["Xq"], p["s_a"], p.get("Xe"))
        ios.append(StarqQuantIo(_p(p["X"]), _p(p.get("mask")), _p(p.get("a_m")), _p(p.get("a_u")), p["d_sh"],
                                p["d_m"], p["d_u"], _p(p["Xq"]), _p(p["s_a"]), _p(p.get("Xe")),
                                int(bool(p.get("independent", False)))))
    L, K = X0.shape
    _check(lib.sgat_quantize_act_grouped(ctypes.byref(ios[0]), ctypes.byref(ios[1]), dtype_code(X0), L, K, hb,
                                         bits, _stream(stream)))


def sgat_prepare_weight(W, inv_a_w, hb, Wq, s_w, bits=4, stream=None):
    _contig(W, inv_a_w, Wq, s_w)
    N, K = W.shape
    _check(lib.sgat_prepare_weight(_p(W), dtype_code(W), N, K, _p(inv_a_w), hb, bits,
                                   _p(Wq), _p(s_w), _stream(stream)))


def _weight_shape(Wq, We):
    if Wq is not None:
        return Wq.shape[0], 2 * Wq.shape[1]
    return We.shape[0], We.shape[1]


def w4_unpack_e4m3(Wq, We, stream=None):
    """Packed int4 weight codes [N][K/2] -> E4M3 bytes [N][K] (once per weight)."""
    _contig(Wq, We)
    N, K = We.shape
    _check(lib.w4_unpack_e4m3(_p(Wq), N, K, _p(We), _stream(stream)))


def sgat_quantize_act_asym(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, Xq, s_a, z_a, Xe=None, stream=None):
    """Asymmetric 4-bit activation codes (Eq. 2-4): Xq [L][K/2] unsigned
    nibbles, s_a [L], z_a [L] int32; Xe [L][K + 128] E4M3 codes + zero-point
    columns."""
    _contig(X, mask, a_m, a_u, Xq, s_a, z_a, Xe)
    L, K = X.shape
    _check(lib.sgat_quantize_act_asym(_p(X), dtype_code(X), L, K, _p(mask), _p(a_m), _p(a_u), hb, d_sh, d_m, d_u,
                                      _p(Xq), _p(s_a), _p(z_a), _p(Xe), _stream(stream)))


def w4_zero_point_columns(Wq, We, stream=None):
    """Packed 4-bit weight codes [N][K/2] -> E4M3 rows [N][K + 128] (codes,
    then 128 values summing to the row's code sum)."""
    _contig(Wq, We)
    N = Wq.shape[0]
    K = We.shape[1] - 128
    _check(lib.w4_zero_point_columns(_p(Wq), N, K, _p(We), _stream(stream)))


def sgat_linear_asym_workspace_size(L, K):
    return int(lib.sgat_linear_asym_workspace_size(L, K))


def sgat_linear_asym(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, We, s_w, Y, workspace, bias=None, stream=None):
    _contig(X, mask, a_m, a_u, We, s_w, Y, workspace, bias)
    L, K = X.shape
    N = We.shape[0]
    _check(lib.sgat_linear_asym(_p(X), dtype_code(X), L, K, _p(mask), _p(a_m), _p(a_u), hb, d_sh, d_m, d_u,
                                _p(We), _p(s_w), _p(bias), N, _p(Y), dtype_code(Y), _p(workspace),
                                workspace.numel() * workspace.element_size(), _stream(stream)))


def _ws(n, device):
    return torch.empty(int(n), dtype=torch.uint8, device=device)


def sgat_quantize_act_dense(X, mask, a_m, a_u, Pt, d_sh, d_m, d_u, Xq, s_a, Xe=None, workspace=None, stream=None):
    """Dense-basis activation codes: Pt = P^T [K][K] float16 (P orthogonal).
    workspace (optional) holds the scaled rows and V = X^s P (float16)."""
    L, K = X.shape
    if workspace is None:
        workspace = _ws(lib.sgat_dense_workspace_size(L, K), X.device)
    _contig(X, mask, a_m, a_u, Pt, Xq, s_a, Xe, workspace)
    _check(lib.sgat_quantize_act_dense(_p(X), dtype_code(X), L, K, _p(mask), _p(a_m), _p(a_u), _p(Pt), d_sh, d_m,
                                       d_u, _p(Xq), _p(s_a), _p(Xe), _p(workspace),
                                       workspace.numel() * workspace.element_size(), _stream(stream)))
    return workspace


def sgat_prepare_weight_dense(W, inv_a_w, Pt, Wq, s_w, workspace=None, stream=None):
    N, K = W.shape
    if workspace is None:
        workspace = _ws(lib.sgat_dense_workspace_size(N, K), W.device)
    _contig(W, inv_a_w, Pt, Wq, s_w, workspace)
    _check(lib.sgat_prepare_weight_dense(_p(W), dtype_code(W), N, K, _p(inv_a_w), _p(Pt), _p(Wq), _p(s_w),
                                         _p(workspace), workspace.numel() * workspace.element_size(),
                                         _stream(stream)))
    return workspace


def sgat_linear_dense_workspace_size(L, K):
    return int(lib.sgat_linear_dense_workspace_size(L, K))


def sgat_linear_dense(X, mask, a_m, a_u, Pt, d_sh, d_m, d_u, Wq, s_w, Y, workspace, bias=None, We=None, stream=None):
    _contig(X, mask, a_m, a_u, Pt, Wq, We, s_w, Y, workspace, bias)
    L, K = X.shape
    N = _weight_shape(Wq, We)[0]
    _check(lib.sgat_linear_dense(_p(X), dtype_code(X), L, K, _p(mask), _p(a_m), _p(a_u), _p(Pt), d_sh, d_m, d_u,
                                 _p(Wq), _p(We), _p(s_w), _p(bias), N, _p(Y), dtype_code(Y), _p(workspace),
                                 workspace.numel() * workspace.element_size(), _stream(stream)))


def w8_codes_f16(Wq, We, stream=None):
    """8-bit weight codes [N][K] (int8) -> the same codes as fp16 [N][K]
    (We: 2K bytes a row, any dtype; once per weight)."""
    _contig(Wq, We)
    N, K = Wq.shape
    _check(lib.w8_codes_f16(_p(Wq), N, K, _p(We), _stream(stream)))


def w8a8_gemm(Xe, s_a, We, s_w, Y, bias=None, acc_dbg=None, stream=None):
    """Xe: activation codes as fp16 [L][K] (sgat_quantize_act with bits=8),
    We: weight codes as fp16 [N][K] (w8_codes_f16), each held as 2K bytes a
    row; Y [L][N]."""
    _contig(Xe, s_a, We, s_w, Y, bias, acc_dbg)
    L, N = Y.shape
    K = We.shape[1] * We.element_size() // 2
    _check(lib.w8a8_gemm(_p(Xe), _p(s_a), _p(We), _p(s_w), _p(bias), L, N, K, _p(Y), dtype_code(Y), _p(acc_dbg),
                         _stream(stream)))


def w4a4_gemm(Xq, s_a, Wq, s_w, Y, bias=None, acc_dbg=None, Xe=None, We=None, stream=None, tac_M=None,
              tac_d=None, tac_g=0, tac_Mp=None, tac_scratch=None):
    """Xq: packed int4 codes [L][K/2] (may be None when Xe is given);
    Xe: the same codes as E4M3 bytes [L][K] (selects a TMA CTA-pair kernel);
    We: the weight codes as E4M3 bytes [N][K] (with Xe: both operands by TMA).
    With tac_M: the dequantised output goes to tac_scratch [L][N] (Y's type)
    and Y receives its TAC."""
    _contig(Xq, Xe, s_a, Wq, We, s_w, Y, bias, acc_dbg)
    L = Y.shape[0]
    N, K = _weight_shape(Wq, We)
    tac = _tac_struct(tac_M, tac_d, tac_g, tac_Mp, tac_scratch)
    _check(lib.w4a4_gemm(_p(Xq), _p(Xe), _p(s_a), _p(Wq), _p(We), _p(s_w), _p(bias), L, N, K, _p(Y),
                         dtype_code(Y), _ref(tac), _p(acc_dbg), _stream(stream)))


GEMM_WEIGHTS_READY = 1


def w4a4_gemm_grouped(Xe0, s_a0, We0, s_w0, Y0, Xe1, s_a1, We1, s_w1, Y1, bias0=None, bias1=None,
                      acc_dbg0=None, acc_dbg1=None, weights_ready=False, stream=None):
    """Two independent W4A4 products (same L, K and output type) in one
    launch: Y0 from Xe0 [L][K] and We0 [N0][K], Y1 from Xe1 and We1 (E4M3
    codes). weights_ready: the launch just before this one does not write
    We0 or We1 (their first tiles are fetched while it finishes)."""
    _contig(Xe0, s_a0, We0, s_w0, Y0, bias0, acc_dbg0, Xe1, s_a1, We1, s_w1, Y1, bias1, acc_dbg1)
    L, K = Xe0.shape
    if tuple(Xe1.shape) != (L, K) or Y0.dtype != Y1.dtype:
        raise StarqError(-2, "w4a4_gemm_grouped: the problems need the same L, K and output type")
    _check(lib.w4a4_gemm_grouped(_p(Xe0), _p(s_a0), _p(We0), _p(s_w0), _p(bias0), We0.shape[0], _p(Y0),
                                 _p(Xe1), _p(s_a1), _p(We1), _p(s_w1), _p(bias1), We1.shape[0], _p(Y1), L, K,
                                 dtype_code(Y0), _p(acc_dbg0), _p(acc_dbg1),
                                 GEMM_WEIGHTS_READY if weights_ready else 0, _stream(stream)))


def w4a4_gemm_mma_sync(Xq, s_a, Wq, s_w, Y, bias=None, acc_dbg=None, stream=None):
    """The same product on the warp-level int4 MMA (mma.sync s4), packed
    operands Xq [L][K/2], Wq [N][K/2]."""
    _contig(Xq, s_a, Wq, s_w, Y, bias, acc_dbg)
    L, N = Y.shape
    K = Wq.shape[1] * 2
    _check(lib.w4a4_gemm_mma_sync(_p(Xq), _p(s_a), _p(Wq), _p(s_w), _p(bias), L, N, K, _p(Y), dtype_code(Y),
                                  _p(acc_dbg), _stream(stream)))


def set_gemm_pair_limit(pairs):
    """Cap the CTA pairs of the pair GEMMs launched afterwards from this
    thread (0 = no cap); returns the previous cap."""
    rc = int(lib.starq_set_gemm_pair_limit(int(pairs)))
    if rc < 0:
        raise StarqError(rc, lib.starq_last_error().decode())
    return rc


def last_gemm_tile():
    """(channels per pair tile, CTAs per cluster) of the calling thread's
    last TMA pair GEMM launch, or None before the first."""
    t = int(lib.starq_last_gemm_tile())
    return (t // 10, t % 10) if t else None


def fp16_gemm_ref(A, B, C, stream=None):
    """C = A B^T for 16-bit A [M][K], B [N][K] (the unquantised baseline)."""
    _contig(A, B, C)
    M, K = A.shape
    N = B.shape[0]
    _check(lib.fp16_gemm_ref(_p(A), _p(B), dtype_code(A), M, N, K, _p(C), _stream(stream)))


def tac_prepare(M, g, z_dtype, Mp, stream=None):
    """M [C/g][g][g] float32 -> the tensor-core form (4 C g bytes) for Z of
    type z_dtype (torch.float16 or torch.bfloat16)."""
    _contig(M, Mp)
    C = M.shape[0] * g
    code = {torch.float16: F16, torch.bfloat16: BF16}[z_dtype]
    _check(lib.tac_prepare(_p(M), C, g, code, _p(Mp), _stream(stream)))


def tac_prepared_bytes(C, g):
    return 4 * C * g


def tac_apply(Z, M, d, g, out, Mp=None, stream=None):
    _contig(Z, M, d, out, Mp)
    L, C = Z.shape
    _check(lib.tac_apply(_p(Z), dtype_code(Z), L, C, g, _p(M), _p(d), _p(Mp), _p(out), dtype_code(out),
                         _stream(stream)))


def tac_calibrate_workspace_size(C, g):
    return int(lib.tac_calibrate_workspace_size(C, g))


def tac_calibrate(Z_fp, Z_q, g, M, d, workspace=None, rho=3e-4, eps=1e-8, eta=0.15, alpha=0.55, stream=None):
    """Closed-form TAC parameters (App. C) from paired calibration outputs
    Z_fp, Z_q [N][C] into M [C/g][g][g] and d [C/g][g] (float32)."""
    _contig(Z_fp, Z_q, M, d, workspace)
    N, C = Z_fp.shape
    assert Z_q.shape == Z_fp.shape and Z_q.dtype == Z_fp.dtype
    if workspace is None:
        workspace = torch.empty(tac_calibrate_workspace_size(C, g), dtype=torch.uint8, device=Z_fp.device)
    _check(lib.tac_calibrate(_p(Z_fp), _p(Z_q), dtype_code(Z_fp), N, C, g, rho, eps, eta, alpha, _p(M), _p(d),
                             _p(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))


def attention_pv_tac_workspace_size(L, Hkv):
    return int(lib.attention_pv_tac_workspace_size(L, Hkv))


def attention_pv_tac(Q, K, V, H, Mp, d, Z, workspace=None, dbg_codes=None, dbg_l=None, dbg_acc=None, Hkv=None,
                     stream=None):
    """Quantised softmax-value product with TAC in its epilogue. Q, K, V are
    fp16 or bf16 [L][ld] views (e.g. column slices of the QKV output) with H
    query heads in Q and Hkv (default H) key/value heads in K and V;
    Z [L][128 H] of the same type."""
    L = Q.shape[0]
    ld = Q.stride(0)
    assert K.stride(0) == ld and V.stride(0) == ld and Q.stride(1) == K.stride(1) == V.stride(1) == 1
    assert Q.dtype == K.dtype == V.dtype == Z.dtype
    Hkv = H if Hkv is None else Hkv
    _contig(Mp, d, Z, workspace, dbg_codes, dbg_l, dbg_acc)
    if workspace is None:
        workspace = torch.empty(attention_pv_tac_workspace_size(L, Hkv), dtype=torch.uint8, device=Q.device)
    _check(lib.attention_pv_tac_gqa(_p(Q), _p(K), _p(V), ld, L, H, Hkv, dtype_code(Q), _p(Mp), _p(d), _p(Z),
                                    _p(dbg_codes), _p(dbg_l), _p(dbg_acc), _p(workspace),
                                    workspace.numel() * workspace.element_size(), _stream(stream)))


def sgat_linear_workspace_size(L, K, with_tac, bits=4):
    if bits == 4:
        return int(lib.sgat_linear_workspace_size(L, K, 1 if with_tac else 0))
    return int(lib.sgat_linear_workspace_size_bits(L, K, 1 if with_tac else 0, bits))


def sgat_linear(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, Wq, s_w, Y, workspace, bias=None,
                tac_M=None, tac_d=None, tac_g=0, bits=4, We=None, tac_Mp=None, stream=None):
    _contig(X, mask, a_m, a_u, Wq, We, s_w, Y, workspace, bias, tac_M, tac_d, tac_Mp)
    L, K = X.shape
    N = _weight_shape(Wq, We)[0]
    _check(lib.sgat_linear(_p(X), dtype_code(X), L, K, _p(mask), _p(a_m), _p(a_u), hb, d_sh, d_m,
                           d_u, _p(tac_M), _p(tac_d), tac_g, _p(tac_Mp), _p(Wq), _p(We), _p(s_w), _p(bias), N, bits,
                           _p(Y), dtype_code(Y), _p(workspace), workspace.numel() * workspace.element_size(),
                           _stream(stream)))


def swiglu_row_order(F, device="cpu"):
    """Row order of a gate+up weight [2F][K] (gate rows 0..F-1, up rows
    F..2F-1) for sgat_linear_swiglu: groups of 16 gate rows, each followed by
    the matching 16 up rows."""
    assert F % 16 == 0
    g = torch.arange(F, device=device).view(-1, 16)
    return torch.stack([g, g + F], dim=1).reshape(-1)


def sgat_linear_swiglu(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, Wq, s_w, H, workspace, bias=None,
                       tac_M=None, tac_d=None, tac_g=0, bits=4, We=None, tac_Mp=None, stream=None):
    """sgat_linear with silu(gate) * up fused into the GEMM epilogue: the
    weights' rows in swiglu_row_order, H [L][N / 2]."""
    _contig(X, mask, a_m, a_u, Wq, We, s_w, H, workspace, bias, tac_M, tac_d, tac_Mp)
    L, K = X.shape
    N = _weight_shape(Wq, We)[0]
    _check(lib.sgat_linear_swiglu(_p(X), dtype_code(X), L, K, _p(mask), _p(a_m), _p(a_u), hb, d_sh, d_m,
                                  d_u, _p(tac_M), _p(tac_d), tac_g, _p(tac_Mp), _p(Wq), _p(We), _p(s_w), _p(bias),
                                  N, bits, _p(H), dtype_code(H), _p(workspace),
                                  workspace.numel() * workspace.element_size(), _stream(stream)))


def add_rmsnorm(X, w, Y, R=None, h_out=None, eps=1e-6, stream=None):
    """Y = RMSNorm(X + R) * w (R optional); h_out receives X + R."""
    _contig(X, R, w, h_out, Y)
    L, K = X.shape
    _check(lib.glue_add_rmsnorm(_p(X), _p(R), dtype_code(X), L, K, _p(w), float(eps), _p(h_out), _p(Y),
                                _stream(stream)))


def rope(QK, heads, pos, theta, stream=None):
    """Rotary embedding in place on the first `heads` 128-channel heads of
    each row of QK (a [L][ld] view with unit column stride)."""
    assert QK.stride(1) == 1
    L = QK.shape[0]
    _check(lib.glue_rope(_p(QK), dtype_code(QK), L, QK.stride(0), heads, _p(pos), float(theta), _stream(stream)))


NOALLOC_SCRATCH_BYTES = 32 << 20


def sgat_linear_noalloc(X, mask, a_m, a_u, hb, d_sh, d_m, d_u, Wq, s_w, Y, bias=None,
                        tac_M=None, tac_d=None, tac_g=0, bits=4, We=None, tac_Mp=None, stream=None):
    """sgat_linear without a workspace: the library's fixed device scratch
    array holds the intermediates (see include/starq.h)."""
    _contig(X, mask, a_m, a_u, Wq, We, s_w, Y, bias, tac_M, tac_d, tac_Mp)
    L, K = X.shape
    N = _weight_shape(Wq, We)[0]
    _check(lib.sgat_linear_noalloc(_p(X), dtype_code(X), L, K, _p(mask), _p(a_m), _p(a_u), hb, d_sh,
                                   d_m, d_u, _p(tac_M), _p(tac_d), tac_g, _p(tac_Mp), _p(Wq), _p(We), _p(s_w), _p(bias), N,
                                   bits, _p(Y), dtype_code(Y), _stream(stream)))
