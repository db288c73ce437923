"""Shared test plumbing: device transfer, oracle runs, tolerances.

Tolerances:
  * int codes, scales and integer accumulators: bit-exact.
  * dequantised outputs in float16: |gpu - ref| <= 1e-3 |ref| + 2^-25 (the
    absolute half-spacing of float16 subnormals), ref = float64 oracle.
  * bfloat16 outputs: one bfloat16 rounding alone exceeds 1e-3, so the bound
    is 1e-3 |ref| + half a bfloat16 spacing at max(|ref|, |gpu|): the
    rounding error is bounded by the spacing of the binade the rounded value
    lands in, which can be the one above |ref|'s when ref sits just below a
    power of two.
  * float32 outputs: 1e-6 |ref| + 1e-30.
  * TAC outputs: |gpu - ref| / max(|ref|, 1e-2 rms(ref)) <= 1e-3 (plus the
    output type's half-spacing for 16-bit outputs).
"""

import numpy as np
import torch

from oracle import sgat as osg

F32 = np.float32


def dev(x, dtype=None):
    """numpy -> contiguous CUDA tensor (bf16 values stored as float32 are cast
    exactly)."""
    t = torch.from_numpy(np.ascontiguousarray(x))
    if dtype is not None:
        t = t.to(dtype)
    return t.cuda()


def torch_dtype(name):
    return {"f16": torch.float16, "bf16": torch.bfloat16, "f32": torch.float32}[name]


def host(t):
    return t.detach().float().cpu().numpy() if t.dtype in (torch.float16, torch.bfloat16) else t.detach().cpu().numpy()


def unpack(t):
    return osg.unpack_int4(t.cpu().numpy())


def half_spacing(ref, dtype):
    a = np.abs(ref).astype(np.float64)
    if dtype == "f16":
        return np.full_like(a, 2.0 ** -25)
    if dtype == "bf16":
        e = np.floor(np.log2(np.maximum(a, 2.0 ** -126)))
        return 0.5 * 2.0 ** (e - 7)
    return np.zeros_like(a)


def assert_output_close(gpu, ref, dtype, what="Y"):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert gpu.shape == ref.shape
    if dtype == "f32":
        tol = 1e-6 * np.abs(ref) + 1e-30
    else:
        # one rounding of a value near ref: half a spacing of the binade of the
        # rounded value, which may sit one binade above ref's (hence max)
        tol = 1e-3 * np.abs(ref) + half_spacing(np.maximum(np.abs(ref), np.abs(gpu)), dtype)
        if dtype == "f16":
            tol = 1e-3 * np.abs(ref) + 2.0 ** -25
    err = np.abs(gpu - ref)
    bad = err > tol
    if bad.any():
        i = np.unravel_index(np.argmax(err - tol), err.shape)
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside tolerance; worst at {i}: "
                             f"gpu={gpu[i]!r} ref={ref[i]!r} tol={tol[i]!r}")


def assert_tac_close(gpu, ref, dtype="f32"):
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    floor = 1e-2 * np.sqrt(np.mean(ref ** 2)) if ref.size else 0.0
    denom = np.maximum(np.abs(ref), floor)
    mag = np.maximum(np.abs(ref), np.abs(gpu))     # binade of the rounded value (see assert_output_close)
    err = np.abs(gpu - ref) - half_spacing(mag, dtype) if dtype != "f32" else np.abs(gpu - ref)
    rel = np.max(np.maximum(err, 0) / denom) if ref.size else 0.0
    assert rel <= 1e-3, f"TAC max relative error {rel:.3e} > 1e-3"


def gemm_codes(seed, L, N, K, lo=-7, hi=7):
    rng = np.random.default_rng(seed)
    qa = rng.integers(lo, hi + 1, (L, K)).astype(np.int32)
    qw = rng.integers(lo, hi + 1, (N, K)).astype(np.int32)
    s_a = rng.uniform(0.01, 2.0, L).astype(F32)
    s_w = rng.uniform(0.001, 0.05, N).astype(F32)
    return qa, qw, s_a, s_w


def workspace_views(ws, L, K, with_tac, x_dtype=torch.float32):
    """Views of the intermediates sgat_linear leaves in its workspace
    (the packed-code region, which it leaves unwritten, per-token scales,
    E4M3 codes, the TAC output in the input's type x_dtype), following the
    layout documented for sgat_linear in include/starq.h."""
    a256 = lambda x: (x + 255) // 256 * 256
    o1 = a256(L * K // 2)
    o2 = o1 + a256(4 * L)
    o3 = o2 + a256(L * K)
    Xq = ws[: L * K // 2].view(L, K // 2)
    s_a = ws[o1: o1 + 4 * L].view(torch.float32)
    Xe = ws[o2: o2 + L * K].view(L, K)
    esz = torch.empty(0, dtype=x_dtype).element_size()
    zt = ws[o3: o3 + esz * L * K].view(x_dtype).view(L, K) if with_tac else None
    return Xq, s_a, Xe, zt


def codes_from_e4m3(b):
    """Integer codes in [-8, 8] back from their E4M3 bytes (the inverse of
    e4m3_bytes on its range); any other byte fails the check."""
    b = np.asarray(b.cpu().numpy() if hasattr(b, "cpu") else b, dtype=np.uint8)
    lut = np.full(256, 127, dtype=np.int32)
    q = np.arange(-8, 9)
    lut[e4m3_bytes(q)] = q
    out = lut[b]
    assert np.all(out != 127), "bytes that are not the E4M3 of a code in [-8, 8]"
    return out


def e4m3_bytes(q):
    """E4M3 encoding (1 sign, 4 exponent bits with bias 7, 3 mantissa bits) of
    integer codes in [-8, 8], written from the format's definition:
    |q| = 2^e (1 + m/8) gives byte = sign << 7 | (e + 7) << 3 | m."""
    q = np.asarray(q, dtype=np.int64)
    a = np.abs(q)
    e = np.where(a > 0, np.floor(np.log2(np.maximum(a, 1))).astype(np.int64), 0)
    m = np.where(a > 0, (a * 8 // (1 << e)) - 8, 0)
    b = np.where(a > 0, ((e + 7) << 3) | m, 0)
    return (b | np.where(q < 0, 0x80, 0)).astype(np.uint8)
