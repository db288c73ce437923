"""The full Dream-7B-shaped block (Qwen2.5-7B shape: hidden 3584, 28 query
heads over 4 key/value heads, FFN 18944, bf16, 4 sequences x 2048 tokens,
seeded low-confidence remasking) through the C ABI, every stage checked
against the oracle with teacher forcing (each stage's oracle takes the
GPU's own input to that stage):

- RMSNorm outputs within 1e-3 relative plus half a bf16 spacing;
- every quantised linear: activation codes, scales and E4M3 bytes bit-exact
  with the oracle's state-guided quantiser; outputs within the output
  tolerance of the oracle's dequantised integer GEMM (with the QKV bias;
  silu(gate) * up for the gate/up projection);
- RoPE within half a bf16 spacing plus 1e-5 of the pair's norm;
- grouped-query attention with TAC: the block's output equals a standalone
  call on the same inputs bit for bit, and that call's P codes, integer
  sums and TAC output match the oracle (for sampled heads of one sequence);
- residual sums fl_bf16(a + b) bit-exact.
Rows are sampled (64 across the four sequences, including the masked and
unmasked tokens of each); codes and scales of the sampled rows are exact.
"""

import numpy as np
import pytest
import torch

from oracle import attention as oatt
from oracle import glue as og
from oracle import sgat as osg
from paper_2606_04945_gb300 import inputs
from tests import helpers as H

pytestmark = pytest.mark.gpu
D = 128


def _check_linear(lin, X_rows, mask_rows, rows, Y_rows, L, what, swiglu=False, bias=None):
    xf = lin.xf
    Xq, s_a, Xe, _ = H.workspace_views(lin.workspace, L, lin.K, False)
    codes, s = osg.sgat_quantize_act(X_rows, mask_rows, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, 4)
    assert np.array_equal(H.codes_from_e4m3(Xe)[rows], codes), f"{what}: activation codes"
    assert np.array_equal(s_a.cpu().numpy()[rows], s), f"{what}: activation scales"
    assert np.array_equal(Xe.cpu().numpy()[rows], H.e4m3_bytes(codes)), f"{what}: E4M3 codes"
    ref = osg.dequant(osg.int_gemm(codes, H.unpack(lin.Wq)), s, lin.s_w.cpu().numpy(), bias)
    if swiglu:                                        # rows interleaved by 16: silu(gate) * up
        r = ref.reshape(len(rows), -1, 2, 16)
        ref = og.swiglu(r[:, :, 0, :].reshape(len(rows), -1), r[:, :, 1, :].reshape(len(rows), -1))
    H.assert_output_close(Y_rows, ref, "bf16", what=what)


def test_dream_block(abi):
    from paper_2606_04945_gb300.dream import DreamBlock
    case = inputs.dream_block(seed=0)
    blk = DreamBlock(case)
    got = {}
    out = blk.forward(hook=lambda name, t: got.__setitem__(name, H.host(t)))
    abi.check_status()
    out = H.host(out)
    L, S = case.L, case.seq
    rng = np.random.default_rng(1)
    rows = []
    for b in range(case.batch):
        m = np.nonzero(case.mask[b * S:(b + 1) * S])[0]
        u = np.nonzero(case.mask[b * S:(b + 1) * S] == 0)[0]
        rows += list(b * S + rng.choice(m, 6, replace=False)) + list(b * S + rng.choice(u, 10, replace=False))
    rows = np.unique(np.array(rows + [0, L - 1]))
    mrows = case.mask[rows]
    X = case.X

    # pre-norm
    H.assert_output_close(got["a"][rows], og.rmsnorm(X[rows], case.w_ln1, case.eps), "bf16", what="RMSNorm 1")
    # QKV with bias
    _check_linear(blk.qkv, got["a"][rows], mrows, rows, got["qkv"][rows], L, "QKV", bias=case.b_qkv)
    # RoPE on the 32 query and key heads
    nrot = case.heads + case.kv_heads
    f32 = og.rope_frequencies(case.rope_theta).astype(np.float32)
    ang = case.pos[rows].astype(np.float32)[:, None] * f32[None, :]
    ref = og.rope(got["qkv"][rows], case.pos[rows], nrot, case.rope_theta, angles=ang)
    pre = got["qkv"][rows].astype(np.float64)
    a, b_ = pre[:, :nrot * D].reshape(len(rows), nrot, 2, 64)[:, :, 0], pre[:, :nrot * D].reshape(len(rows), nrot, 2, 64)[:, :, 1]
    norm = np.repeat(np.sqrt(a * a + b_ * b_)[:, :, None, :], 2, axis=2).reshape(len(rows), nrot * D)
    rot = got["qkv_rope"][rows].astype(np.float64)
    assert np.all(np.abs(rot[:, :nrot * D] - ref[:, :nrot * D]) <= H.half_spacing(ref[:, :nrot * D], "bf16") + 1e-5 * norm)
    assert np.array_equal(rot[:, nrot * D:], pre[:, nrot * D:])

    # attention of sequence 0: the block's output against a standalone call
    # with the debug outputs, and that call against the oracle
    Cq, Ckv = case.heads * D, case.kv_heads * D
    qkv0 = torch.from_numpy(got["qkv_rope"][:S]).to(torch.bfloat16).cuda()
    Z = torch.empty(S, Cq, dtype=torch.bfloat16, device="cuda")
    codes = torch.zeros(case.heads, S, S, dtype=torch.uint8, device="cuda")
    lsum = torch.zeros(case.heads, S, dtype=torch.float32, device="cuda")
    acc = torch.zeros(case.heads, S, D, dtype=torch.int32, device="cuda")
    abi.attention_pv_tac(qkv0[:, :Cq], qkv0[:, Cq:Cq + Ckv], qkv0[:, Cq + Ckv:], case.heads, blk.tac_Mp, blk.tac_d, Z,
                         dbg_codes=codes, dbg_l=lsum, dbg_acc=acc, Hkv=case.kv_heads)
    abi.check_status()
    assert np.array_equal(H.host(Z), got["z"][:S])
    Qn, Kn, Vn = got["qkv_rope"][:S, :Cq], got["qkv_rope"][:S, Cq:Cq + Ckv], got["qkv_rope"][:S, Cq + Ckv:]
    vq, t = oatt.v_codes(Vn)
    gcodes, gl, gacc = codes.cpu().numpy().astype(np.int32), lsum.cpu().numpy(), acc.cpu().numpy()
    group = case.heads // case.kv_heads
    for h in (0, 6, 7, 20, 27):
        ch, kv = slice(h * D, (h + 1) * D), slice((h // group) * D, (h // group + 1) * D)
        Sc = oatt.scores(Qn[:, ch], Kn[:, kv], D)
        oc, ol = oatt.p_codes(Sc)
        diff = gcodes[h] != oc
        if diff.any():
            e255 = 255.0 * np.exp(Sc - Sc.max(axis=1, keepdims=True))
            near = np.abs(e255 - np.floor(e255) - 0.5) < 1e-3
            assert np.all(np.abs(gcodes[h] - oc)[diff] == 1) and np.all(near[diff]), f"head {h}: P codes"
        np.testing.assert_allclose(gl[h], ol, rtol=1e-5)
        ref_acc = osg.int_gemm(gcodes[h], vq[:, kv].T)
        assert np.array_equal(gacc[h], ref_acc), f"head {h}: integer sums"
        zhat = ref_acc.astype(np.float64) / (255.0 * gl[h].astype(np.float64)[:, None]) * t[kv].astype(np.float64)
        refz = zhat @ case.tac.M[h].astype(np.float64).T + case.tac.d[h].astype(np.float64)[None, :]
        H.assert_tac_close(got["z"][:S, ch], refz, "bf16")
    del codes

    # O projection, residual and the second norm
    _check_linear(blk.o, got["z"][rows], mrows, rows, got["o"][rows], L, "O")
    x1 = inputs.round_to_bf16(X[rows] + got["o"][rows])
    assert np.array_equal(got["x1"][rows], x1)
    H.assert_output_close(got["a2"][rows], og.rmsnorm(x1, case.w_ln2, case.eps), "bf16", what="RMSNorm 2")
    # gate/up with SwiGLU, down, final residual
    _check_linear(blk.gu, got["a2"][rows], mrows, rows, got["g"][rows], L, "gate/up", swiglu=True)
    _check_linear(blk.down, got["g"][rows], mrows, rows, got["d"][rows], L, "down")
    assert np.array_equal(out[rows], inputs.round_to_bf16(got["x1"][rows] + got["d"][rows]))
    assert np.all(np.isfinite(out))
