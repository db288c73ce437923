"""The LLaDA attention-projection step as the bench runs it, in both of its
forms: forked (the QKV projection on the calling stream, TAC + O projection
on a side stream, joined inside one CUDA graph) and grouped (the two
quantisations on two streams, then both GEMMs in one w4a4_gemm_grouped
launch). Its outputs must equal those of the two projections run one after
the other on one stream (which the parity tests check against the oracle),
eagerly and on graph replay, and the step's buffers must not be touched by a
replay of the other branch.
"""

import pytest
import torch

from paper_2606_04945_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("grouped", [False, "gemm", True])
def test_step_equals_sequential(abi, grouped):
    from paper_2606_04945_gb300.pipeline import AttentionProjections
    qkv_case, o_case = inputs.llada_attention(seed=3)
    st = AttentionProjections(qkv_case, o_case, grouped=grouped)
    assert st.KERNELS_PER_STEP == {False: 5, "gemm": 4, True: 3}[grouped]
    st.qkv.run(st.X, st.mask, st.Y_qkv)
    st.o.run(st.Z, st.mask, st.Y_o)
    torch.cuda.synchronize()
    ref_q, ref_o = st.Y_qkv.clone(), st.Y_o.clone()

    st.Y_qkv.zero_()
    st.Y_o.zero_()
    st.step()
    torch.cuda.synchronize()
    abi.check_status()
    assert torch.equal(st.Y_qkv, ref_q)
    assert torch.equal(st.Y_o, ref_o)

    st.capture()
    for _ in range(3):
        st.Y_qkv.zero_()
        st.Y_o.zero_()
        st.replay()
        torch.cuda.synchronize()
        assert torch.equal(st.Y_qkv, ref_q)
        assert torch.equal(st.Y_o, ref_o)
    abi.check_status()
