"""Glue kernels of the quantised blocks (residual add + RMSNorm, rotary
embedding) against oracle/glue.py.

- The residual sum h = fl_T(x + r) is one float32 addition of two 16-bit
  values and one rounding: bit-exact.
- RMSNorm, teacher-forced on the GPU's h (float32 sum of squares and
  rsqrtf against float64): within 1e-3 relative plus half a spacing of the
  output type.
- Rotary embedding with the kernel's float32 angles fl(pos * fl32(f_i)):
  within half a spacing of the output type plus 1e-5 of the pair's norm
  (float32 trigonometry and products).
"""

import numpy as np
import pytest
import torch

from oracle import glue as og
from paper_2606_04945_gb300 import inputs
from tests import helpers as H

pytestmark = pytest.mark.gpu


def _round(x, dt):
    return x.astype(np.float16).astype(np.float32) if dt == "f16" else inputs.round_to_bf16(x)


def _half_ulp(ref, dt):
    """Half a spacing of the output type at |ref| (one rounding)."""
    if dt == "f16":
        return 2.0 ** -11 * np.abs(ref) + 2.0 ** -25
    return H.half_spacing(ref, dt)


@pytest.mark.parametrize("L,K,dt,resid", [(37, 3584, "bf16", True), (64, 4096, "f16", False), (5, 18944, "bf16", True)])
def test_add_rmsnorm(abi, L, K, dt, resid):
    rng = np.random.default_rng(L + K)
    x = _round(rng.normal(0, 1, (L, K)).astype(np.float32) * 3, dt)
    r = _round(rng.normal(0, 1, (L, K)).astype(np.float32), dt) if resid else None
    w = rng.normal(1, 0.2, K).astype(np.float32)
    tdt = H.torch_dtype(dt)
    X = H.dev(x, tdt)
    R = H.dev(r, tdt) if resid else None
    Hout = torch.empty_like(X) if resid else None
    Y = torch.empty_like(X)
    abi.add_rmsnorm(X, H.dev(w), Y, R=R, h_out=Hout, eps=1e-6)
    torch.cuda.synchronize()
    if resid:
        h = H.host(Hout)
        assert np.array_equal(h, _round(x + r, dt))            # float32 sum, one rounding
    else:
        h = x
    ref = og.rmsnorm(h, w, 1e-6)
    got = H.host(Y).astype(np.float64)
    assert np.all(np.abs(got - ref) <= 1e-3 * np.abs(ref) + H.half_spacing(ref, dt) + 1e-6)


def test_add_rmsnorm_in_place(abi):
    """h_out = R (the residual stream updated in place)."""
    rng = np.random.default_rng(9)
    x = _round(rng.normal(0, 1, (8, 1024)).astype(np.float32), "bf16")
    r = _round(rng.normal(0, 1, (8, 1024)).astype(np.float32), "bf16")
    X, R = H.dev(x, torch.bfloat16), H.dev(r, torch.bfloat16)
    abi.add_rmsnorm(X, H.dev(np.ones(1024, np.float32)), torch.empty_like(X), R=R, h_out=R)
    torch.cuda.synchronize()
    assert np.array_equal(H.host(R), _round(x + r, "bf16"))


@pytest.mark.parametrize("L,heads,extra,dt", [(300, 32, 512, "bf16"), (128, 4, 0, "f16")])
def test_rope(abi, L, heads, extra, dt):
    rng = np.random.default_rng(L + heads)
    C = heads * 128 + extra
    x = _round(rng.normal(0, 1, (L, C)).astype(np.float32), dt)
    pos = rng.integers(0, 2048, L).astype(np.int32)
    tdt = H.torch_dtype(dt)
    QK = H.dev(x, tdt)
    abi.rope(QK, heads, H.dev(pos), 1e6)
    torch.cuda.synchronize()
    f32 = og.rope_frequencies(1e6).astype(np.float32)
    ang = pos.astype(np.float32)[:, None] * f32[None, :]          # float32 products, as the kernel
    ref = og.rope(x, pos, heads, 1e6, angles=ang)
    got = H.host(QK).astype(np.float64)
    norm = np.zeros_like(ref)
    for h in range(heads):
        a, b = x[:, h * 128:h * 128 + 64].astype(np.float64), x[:, h * 128 + 64:(h + 1) * 128].astype(np.float64)
        n = np.sqrt(a * a + b * b)
        norm[:, h * 128:h * 128 + 64] = n
        norm[:, h * 128 + 64:(h + 1) * 128] = n
    assert np.all(np.abs(got - ref) <= _half_ulp(ref, dt) + 1e-5 * norm)
    assert np.array_equal(got[:, heads * 128:], x[:, heads * 128:])
