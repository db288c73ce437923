"""attention_pv_tac: the quantised softmax-value product with TAC fused into
its dequantisation epilogue, against the oracle (oracle/attention.py).

Q, K and V are the three column slices of one fp16 [L][3 * 128 H] QKV
output (the layout the QKV projection writes), N(0, 1). The TAC blocks
are I + N(0, 0.01), one per head. The comparisons:

- P codes at every position. The kernel takes exp in float32 (the PTX
  approximation, relative error about 2^-22, so 255 e to about 1e-4) and
  the oracle in float64, so a code may differ by one, but only where 255 e
  lies within 1e-3 of a half-integer (the decision is a floating-point
  rounding; elsewhere the codes are equal);
- row sums l to 1e-5 relative;
- the exact integer sums, bit for bit, against the oracle's integer product
  of the GPU's P codes and the oracle's V codes. This pins the V codes and
  the P V^T contraction exactly;
- the TAC output, teacher-forced on the GPU's codes and sums, within the
  TAC tolerance (1e-3 relative, fp16 output).
"""

import numpy as np
import pytest
import torch

from oracle import attention as oatt
from oracle import sgat as osg
from oracle import tac as otac
from paper_2606_04945_gb300 import inputs
from tests import helpers as H

pytestmark = pytest.mark.gpu
D = 128


def run_case(abi, L, Hh, seed, heads=None, zero_q=False, v_signs=None):
    """v_signs: per-channel signs [128 H]; V is then +-1 down each column,
    so every V code is +-7."""
    rng = np.random.default_rng(seed)
    C = D * Hh
    QKV = rng.standard_normal((L, 3 * C)).astype(np.float16)
    if zero_q:
        QKV[:, :C] = 0
    if v_signs is not None:
        QKV[:, 2 * C:] = np.broadcast_to(np.asarray(v_signs, np.float16)[None, :], (L, C))
    Y = torch.from_numpy(QKV).cuda()
    Q, K, V = Y[:, :C], Y[:, C:2 * C], Y[:, 2 * C:]
    tac = inputs.make_tac(rng, C, D)
    M, dvec = H.dev(tac.M), H.dev(tac.d)
    Mp = torch.empty(abi.tac_prepared_bytes(C, D), dtype=torch.uint8, device="cuda")
    abi.tac_prepare(M, D, torch.float16, Mp)
    Z = torch.full((L, C), float("nan"), dtype=torch.float16, device="cuda")
    codes = torch.zeros(Hh, L, L, dtype=torch.uint8, device="cuda")
    lsum = torch.zeros(Hh, L, dtype=torch.float32, device="cuda")
    acc = torch.zeros(Hh, L, D, dtype=torch.int32, device="cuda")
    abi.attention_pv_tac(Q, K, V, Hh, Mp, dvec, Z, dbg_codes=codes, dbg_l=lsum, dbg_acc=acc)
    abi.check_status()
    Zg = H.host(Z)
    assert not np.isnan(Zg).any()
    gcodes, gl, gacc = codes.cpu().numpy().astype(np.int32), lsum.cpu().numpy(), acc.cpu().numpy()
    Qn, Kn, Vn = (QKV[:, i * C:(i + 1) * C].astype(np.float32) for i in range(3))
    vq, t = oatt.v_codes(Vn)
    for h in (range(Hh) if heads is None else heads):
        ch = slice(h * D, (h + 1) * D)
        S = oatt.scores(Qn[:, ch], Kn[:, ch], D)
        oc, ol = oatt.p_codes(S)
        diff = gcodes[h] != oc
        if diff.any():
            e255 = 255.0 * np.exp(S - S.max(axis=1, keepdims=True))
            near = np.abs(e255 - np.floor(e255) - 0.5) < 1e-3
            assert np.all(np.abs(gcodes[h] - oc)[diff] == 1) and np.all(near[diff]), f"head {h}: P codes"
        np.testing.assert_allclose(gl[h], ol, rtol=1e-5, err_msg=f"head {h}: row sums")
        ref_acc = osg.int_gemm(gcodes[h], vq[:, ch].T)
        assert np.array_equal(gacc[h], ref_acc), f"head {h}: integer sums"
        zhat = ref_acc.astype(np.float64) / (255.0 * gl[h].astype(np.float64)[:, None]) * t[ch].astype(np.float64)
        ref = zhat @ tac.M[h].astype(np.float64).T + tac.d[h].astype(np.float64)[None, :]
        H.assert_tac_close(Zg[:, ch], ref, "f16")
    return Zg, gcodes, t, vq, tac


@pytest.mark.parametrize("L,Hh", [(128, 1), (256, 2), (640, 3)])
def test_attention_pv_tac_matches_oracle(abi, L, Hh):
    run_case(abi, L, Hh, seed=L + Hh)


def test_attention_pv_tac_llada_width(abi):
    """1024 tokens, 32 heads of 128 (the LLaDA-8B attention width): every
    head checked against the oracle."""
    run_case(abi, 1024, 32, seed=11)


@pytest.mark.parametrize("L,Hh", [(2048, 2), (8192, 1)])
def test_attention_pv_tac_long(abi, L, Hh):
    """The Dream-7B sequence length (2048) and the longest supported one
    (8192): 16 and 64 key chunks per query tile, every head checked."""
    run_case(abi, L, Hh, seed=L + 7 * Hh)


def test_attention_pv_tac_exact_at_2_24_edge(abi):
    """The largest integer sums the kernel can meet: L = 8192 with Q = 0
    (every P code 255) and V = +-1 down each channel (every V code +-7), so
    acc = +-255 * 7 * 8192 = +-14,622,720, just below 2^24 = 16,777,216
    where float32 would stop holding every integer. The sums must come back
    exact, and Z_hat = acc / (255 l) * t = +-1 before TAC."""
    L, Hh = 8192, 1
    signs = np.where(np.random.default_rng(5).random(D * Hh) < 0.5, -1.0, 1.0)
    rng = np.random.default_rng(9)
    C = D * Hh
    QKV = np.zeros((L, 3 * C), np.float16)
    QKV[:, C:2 * C] = rng.standard_normal((L, C)).astype(np.float16)
    QKV[:, 2 * C:] = np.broadcast_to(signs.astype(np.float16)[None, :], (L, C))
    Y = torch.from_numpy(QKV).cuda()
    tac = inputs.make_tac(rng, C, D)
    Mp = torch.empty(abi.tac_prepared_bytes(C, D), dtype=torch.uint8, device="cuda")
    abi.tac_prepare(H.dev(tac.M), D, torch.float16, Mp)
    Z = torch.full((L, C), float("nan"), dtype=torch.float16, device="cuda")
    acc = torch.zeros(Hh, L, D, dtype=torch.int32, device="cuda")
    lsum = torch.zeros(Hh, L, dtype=torch.float32, device="cuda")
    abi.attention_pv_tac(Y[:, :C], Y[:, C:2 * C], Y[:, 2 * C:], Hh, Mp, H.dev(tac.d), Z, dbg_l=lsum, dbg_acc=acc)
    abi.check_status()
    expect = (255 * 7 * L) * signs.astype(np.int64)
    assert 255 * 7 * L == 14622720 < 2 ** 24
    assert np.array_equal(acc.cpu().numpy()[0], np.broadcast_to(expect[None, :], (L, D)))
    assert np.all(lsum.cpu().numpy() == float(L))                  # exp(0) summed exactly
    zhat = np.broadcast_to(signs[None, :], (L, D)).astype(np.float64)
    ref = zhat @ tac.M[0].astype(np.float64).T + tac.d[0].astype(np.float64)[None, :]
    H.assert_tac_close(H.host(Z), ref, "f16")


def test_attention_pv_tac_uniform(abi):
    """Q = 0: uniform attention, every code 255, and Z = TAC(mean over keys
    of the dequantised V)."""
    L, Hh = 256, 2
    Zg, gcodes, t, vq, tac = run_case(abi, L, Hh, seed=3, zero_q=True)
    assert np.all(gcodes == 255)
    for h in range(Hh):
        ch = slice(h * D, (h + 1) * D)
        mean = (vq[:, ch] * t[ch][None, :]).astype(np.float64).mean(axis=0)
        ref = np.broadcast_to(mean @ tac.M[h].T + tac.d[h], (L, D))
        H.assert_tac_close(Zg[:, ch], ref, "f16")


def run_case_gqa(abi, L, Hh, Hkv, dt, seed, heads=None):
    """Grouped-query case: Q with Hh heads, K and V with Hkv heads, element
    type dt ("f16" or "bf16"); the comparisons of run_case, with query head h
    reading key/value head h // (Hh / Hkv)."""
    rng = np.random.default_rng(seed)
    C, Ckv = D * Hh, D * Hkv
    QKV = rng.standard_normal((L, C + 2 * Ckv)).astype(np.float32)
    QKV = QKV.astype(np.float16).astype(np.float32) if dt == "f16" else inputs.round_to_bf16(QKV)
    tdt = H.torch_dtype(dt)
    Y = H.dev(QKV, tdt)
    Q, K, V = Y[:, :C], Y[:, C:C + Ckv], Y[:, C + Ckv:]
    tac = inputs.make_tac(rng, C, D)
    Mp = torch.empty(abi.tac_prepared_bytes(C, D), dtype=torch.uint8, device="cuda")
    abi.tac_prepare(H.dev(tac.M), D, torch.float16, Mp)      # fp16 halves for either I/O type
    Z = torch.full((L, C), float("nan"), dtype=tdt, device="cuda")
    codes = torch.zeros(Hh, L, L, dtype=torch.uint8, device="cuda")
    lsum = torch.zeros(Hh, L, dtype=torch.float32, device="cuda")
    acc = torch.zeros(Hh, L, D, dtype=torch.int32, device="cuda")
    abi.attention_pv_tac(Q, K, V, Hh, Mp, H.dev(tac.d), Z, dbg_codes=codes, dbg_l=lsum, dbg_acc=acc, Hkv=Hkv)
    abi.check_status()
    Zg = H.host(Z)
    assert not np.isnan(Zg).any()
    gcodes, gl, gacc = codes.cpu().numpy().astype(np.int32), lsum.cpu().numpy(), acc.cpu().numpy()
    Qn, Kn, Vn = QKV[:, :C], QKV[:, C:C + Ckv], QKV[:, C + Ckv:]
    vq, t = oatt.v_codes(Vn)
    group = Hh // Hkv
    for h in (range(Hh) if heads is None else heads):
        ch = slice(h * D, (h + 1) * D)
        kv = slice((h // group) * D, (h // group + 1) * D)
        S = oatt.scores(Qn[:, ch], Kn[:, kv], D)
        oc, ol = oatt.p_codes(S)
        diff = gcodes[h] != oc
        if diff.any():
            e255 = 255.0 * np.exp(S - S.max(axis=1, keepdims=True))
            near = np.abs(e255 - np.floor(e255) - 0.5) < 1e-3
            assert np.all(np.abs(gcodes[h] - oc)[diff] == 1) and np.all(near[diff]), f"head {h}: P codes"
        np.testing.assert_allclose(gl[h], ol, rtol=1e-5, err_msg=f"head {h}: row sums")
        ref_acc = osg.int_gemm(gcodes[h], vq[:, kv].T)
        assert np.array_equal(gacc[h], ref_acc), f"head {h}: integer sums"
        zhat = ref_acc.astype(np.float64) / (255.0 * gl[h].astype(np.float64)[:, None]) * t[kv].astype(np.float64)
        ref = zhat @ tac.M[h].astype(np.float64).T + tac.d[h].astype(np.float64)[None, :]
        H.assert_tac_close(Zg[:, ch], ref, dt)


@pytest.mark.parametrize("L,Hh,Hkv,dt", [(256, 4, 1, "f16"), (384, 6, 2, "bf16"), (256, 2, 2, "bf16")])
def test_attention_pv_tac_gqa_and_bf16(abi, L, Hh, Hkv, dt):
    run_case_gqa(abi, L, Hh, Hkv, dt, seed=L + 10 * Hh + Hkv)


def test_attention_pv_tac_dream_shape(abi):
    """The Dream-7B attention: 2048 tokens (one sequence), 28 query heads
    over 4 key/value heads, bf16; every seventh head checked (one per
    group and the group edges)."""
    run_case_gqa(abi, 2048, 28, 4, "bf16", seed=28, heads=(0, 6, 7, 13, 20, 27))
