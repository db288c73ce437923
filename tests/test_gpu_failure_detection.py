"""Failure detection without a GPU fault: every wait inside the library's
kernels is bounded, and a wait that runs out sets a bit of the device status
word instead of hanging. starq_selftest_wait_timeout makes one such wait run
out on purpose (a barrier that nothing arms, a 2 ms limit); the host reads
the timeout through starq_check_status, and the context keeps working."""

import re

import numpy as np
import pytest
import torch

from oracle import sgat as osg
from paper_2606_04945_gb300 import inputs
from tests import helpers as H

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_is_reported(abi):
    abi.check_status()                                   # nothing pending
    abi.selftest_wait_timeout(2000)
    with pytest.raises(abi.StarqError) as e:
        abi.check_status()
    assert e.value.code == abi.ERR_TIMEOUT
    bits = int(re.search(r"0x([0-9a-f]+)", str(e.value)).group(1), 16)
    assert bits & 0x4, str(e.value)                      # the self-test bit
    abi.check_status()                                   # the word was cleared


def test_context_usable_after_timeout(abi):
    """After a wait has run out, kernels still run and still match the
    oracle (the quantiser on a small case)."""
    abi.selftest_wait_timeout(1000)
    with pytest.raises(abi.StarqError):
        abi.check_status()
    case = inputs.random_linear(31, 64, 512, 128)
    xf = case.xf
    Xq = torch.empty(case.L, case.K // 2, dtype=torch.uint8, device="cuda")
    s_a = torch.empty(case.L, dtype=torch.float32, device="cuda")
    abi.sgat_quantize_act(H.dev(case.X, torch.float16), H.dev(case.mask), H.dev(xf.a_m), H.dev(xf.a_u), xf.hb,
                          xf.d_sh, xf.d_m, xf.d_u, Xq, s_a)
    abi.check_status()
    codes, s_ref = osg.sgat_quantize_act(case.X, case.mask, xf.a_m, xf.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, 4)[:2]
    assert np.array_equal(H.unpack(Xq), codes)
    assert np.array_equal(s_a.cpu().numpy(), s_ref)


def test_selftest_rejects_bad_limit(abi):
    for bad in (0, 100001):
        with pytest.raises(abi.StarqError) as e:
            abi.selftest_wait_timeout(bad)
        assert e.value.code == abi.ERR_ARG
