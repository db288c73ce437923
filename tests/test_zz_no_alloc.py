"""sgat_linear_noalloc: the entry point for callers that cannot allocate.

Callers such as serving runtimes that own the whole device memory pool, or
plugin interfaces that hand an operator only its inputs and outputs, cannot
supply sgat_linear's workspace. sgat_linear_noalloc keeps the intermediates
in the library's fixed device scratch array instead. These tests call it
through the C ABI and check it against sgat_linear with a caller-owned
workspace, on two calls in a row (the scratch keeps the previous call's
contents, which must not leak into the next result). This file is collected
last so that a run stopping at its first failure has already run every
other test.
"""

import ctypes

import numpy as np
import pytest
import torch

from paper_2606_04945_gb300 import inputs
from tests import helpers as H


def _setup(case, e4m3_weights):
    from paper_2606_04945_gb300 import abi
    from paper_2606_04945_gb300.pipeline import SgatLinear
    layer = SgatLinear(case, e4m3_weights=e4m3_weights)
    X = H.dev(case.X, layer.dtype)
    mask = H.dev(case.mask)
    return abi, layer, X, mask


def _run_both(case, e4m3_weights):
    """sgat_linear (the layer's own workspace) and sgat_linear_noalloc on the
    same arguments, including the layer's E4M3 weights and prepared TAC
    matrices when it has them."""
    abi, layer, X, mask = _setup(case, e4m3_weights)
    Y_ref = torch.empty(case.L, case.N, dtype=layer.out_dtype, device="cuda")
    Y_new = torch.full((case.L, case.N), float("nan"), dtype=layer.out_dtype, device="cuda")
    layer.run(X, mask, Y_ref)
    abi.sgat_linear_noalloc(X, mask, layer.a_m, layer.a_u, layer.hb, layer.d_sh, layer.d_m, layer.d_u,
                            layer.Wq, layer.s_w, Y_new, bias=layer.bias, tac_M=layer.tac_M,
                            tac_d=layer.tac_d, tac_g=layer.tac_g, We=layer.We, tac_Mp=layer.tac_Mp)
    abi.check_status()
    return H.host(Y_new), H.host(Y_ref)


@pytest.mark.gpu
def test_noalloc_matches_sgat_linear_twice():
    """Calls in a row with different shapes, states, TAC settings and weight
    forms: each output matches sgat_linear's within the output tolerance,
    and exactly, since the same kernels run on the same arguments.

    - 1024 x 4096 -> 4096 with TAC (g = 128): E4M3 weights (the TMA GEMM,
      its tensor maps on the scratch array) and prepared TAC matrices;
    - 300 x 1024 -> 512, bf16 with bias, E4M3 weights;
    - the same bf16 case from packed weights only (the converting GEMM)."""
    first = inputs.llada_attention(seed=3)[1]
    second = inputs.random_linear(77, 300, 1024, 512, dtype="bf16", bias=True)
    for case, e4m3 in ((first, True), (second, True), (second, False)):
        y_new, y_ref = _run_both(case, e4m3)
        assert not np.isnan(y_new).any()
        H.assert_output_close(y_new, y_ref, case.dtype, what="sgat_linear_noalloc")
        assert np.array_equal(y_new, y_ref)


@pytest.mark.gpu
def test_noalloc_rejects_oversize():
    from paper_2606_04945_gb300 import abi
    K, L = 4096, 2048                                  # with TAC: 46.1 MB > 32 MiB
    assert abi.sgat_linear_workspace_size(L, K, True) > abi.NOALLOC_SCRATCH_BYTES
    X = torch.zeros(L, K, dtype=torch.float16, device="cuda")
    Wq = torch.zeros(256, K // 2, dtype=torch.uint8, device="cuda")
    s_w = torch.ones(256, dtype=torch.float32, device="cuda")
    M = torch.zeros(K // 128, 128, 128, dtype=torch.float32, device="cuda")
    Y = torch.empty(L, 256, dtype=torch.float16, device="cuda")
    with pytest.raises(abi.StarqError) as e:
        abi.sgat_linear_noalloc(X, None, None, None, 4096, K, 0, 0, Wq, s_w, Y, tac_M=M, tac_g=128)
    assert e.value.code == abi.ERR_SHAPE and "scratch" in str(e.value)


def test_noalloc_symbol_and_limit_declared():
    """The entry point and its limit are part of the C ABI (no GPU needed)."""
    from paper_2606_04945_gb300 import abi
    assert hasattr(abi.lib, "sgat_linear_noalloc")
    src = open(H.__file__.replace("tests/helpers.py", "include/starq.h")).read()
    assert "#define STARQ_NOALLOC_SCRATCH_BYTES (32u << 20)" in src
    assert abi.NOALLOC_SCRATCH_BYTES == 32 << 20
    # the documented limits: 22,532 bytes per token at K = 4096 with TAC,
    # 1489 tokens fit and 1490 do not
    assert abi.sgat_linear_workspace_size(1024, 4096, True) == 23072768
    assert abi.sgat_linear_workspace_size(1489, 4096, True) <= abi.NOALLOC_SCRATCH_BYTES
    assert abi.sgat_linear_workspace_size(1490, 4096, True) > abi.NOALLOC_SCRATCH_BYTES
    assert abi.sgat_linear_workspace_size(1170, 4096, True, bits=8) <= abi.NOALLOC_SCRATCH_BYTES
    assert abi.sgat_linear_workspace_size(1171, 4096, True, bits=8) > abi.NOALLOC_SCRATCH_BYTES
    # the size check runs before any CUDA call
    P = ctypes.c_void_p(4096)
    rc = abi.lib.sgat_linear_noalloc(P, 0, 4096, 4096, None, None, None, 4096, 4096, 0, 0, P, None, 128, None,
                                     P, None, P, None, 256, 4, P, 0, None)
    assert rc == abi.ERR_SHAPE
