"""starq_probe_mma: the tensor-core rate probe behind the GEMM roofline's
denominator. Every kind's accumulators must come back exact (integer sums
through the FP8 tensor cores below 2^24, bf16 sums of ones, the integer
mma.sync kinds), and the rates must be positive and ordered as the
instruction kinds are: the FP8 kind at twice the 16-bit kind's
multiply-adds per clock."""

import pytest
import torch

pytestmark = pytest.mark.gpu


def test_probe_kinds_exact_and_rates(abi):
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    cycles = torch.zeros(4 * sms, dtype=torch.int64, device="cuda")
    errors = torch.zeros(1, dtype=torch.int32, device="cuda")
    rate = {}
    for kind in abi.PROBE_KINDS:
        errors.zero_()
        ctas, macs = abi.probe_mma(kind, 512, cycles, errors)
        abi.check_status()
        assert int(errors.item()) == 0, f"kind {kind}: {int(errors.item())} accumulators not exact"
        cyc = cycles[:ctas].double()
        assert float(cyc.min()) > 0
        per_sm = macs * (ctas / sms if kind >= 3 else 1)          # macs_per_cta is per SM
        rate[kind] = per_sm / float(cyc.max())
    assert 0.75 * 2 * rate[2] < rate[0] < 1.25 * 2 * rate[2], rate
    assert 0.75 * rate[0] < rate[1] < 1.25 * rate[0], rate


def test_probe_rejects_bad_arguments(abi):
    t = torch.zeros(4, dtype=torch.int64, device="cuda")
    e = torch.zeros(1, dtype=torch.int32, device="cuda")
    for kind, iters in ((5, 8), (-1, 8), (0, 0), (0, 4096)):
        with pytest.raises(abi.StarqError) as err:
            abi.probe_mma(kind, iters, t, e)
        assert err.value.code == abi.ERR_ARG
