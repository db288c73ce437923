"""Device-resident SGAT W4A4 layers built on the C ABI.

``SgatLinear`` holds one quantised linear on the GPU: the folded int4
weight (Eq. 12, prepared once by ``sgat_prepare_weight``) and, by default,
the same codes as E4M3 bytes for the tensor cores (``w4_unpack_e4m3``), the
two state transforms, optional TAC parameters and a workspace. ``run`` is one call to
``sgat_linear`` (TAC -> state-guided quantisation -> W4A4 GEMM + dequant).

``AttentionProjections`` is the attention-side hot path of one denoising
step of a LLaDA-shaped layer: the fused QKV projection of the layer input,
then TAC on the attention output followed by the O projection (Sec. 3.3: TAC
sits between the softmax-value product and W_o). ``capture`` records the step
in a CUDA graph so a replay issues all five kernels with one launch; the
two projections run as two branches of the graph.
"""

import numpy as np
import torch

from . import abi


def _dev(x, dtype=None, device="cuda"):
    t = torch.from_numpy(np.ascontiguousarray(x))
    if dtype is not None:
        t = t.to(dtype)
    return t.to(device)


TORCH_DTYPE = {"f16": torch.float16, "bf16": torch.bfloat16, "f32": torch.float32}


class SgatLinear:
    def __init__(self, case, device="cuda", out_dtype=None, e4m3_weights=True):
        xf = case.xf
        self.L, self.K, self.N = case.L, case.K, case.N
        self.dtype = TORCH_DTYPE[case.dtype]
        self.out_dtype = TORCH_DTYPE[out_dtype or case.dtype]
        self.hb, self.d_sh, self.d_m, self.d_u = xf.hb, xf.d_sh, xf.d_m, xf.d_u
        self.a_m = _dev(xf.a_m, device=device)
        self.a_u = _dev(xf.a_u, device=device)
        self.bias = _dev(case.bias, device=device) if case.bias is not None else None
        self.tac = case.tac
        self.tac_Mp = None
        if case.tac is not None:
            self.tac_M = _dev(case.tac.M, device=device)
            self.tac_d = _dev(case.tac.d, device=device)
            self.tac_g = case.tac.g
            if self.dtype != torch.float32 and self.tac_g in (64, 128):
                # TAC matrices in the tensor-core form, once
                self.tac_Mp = torch.empty(abi.tac_prepared_bytes(self.K, self.tac_g), dtype=torch.uint8,
                                          device=device)
                abi.tac_prepare(self.tac_M, self.tac_g, self.dtype, self.tac_Mp)
        else:
            self.tac_M = self.tac_d = None
            self.tac_g = 0
        W = _dev(case.W, self.dtype, device)
        self.Wq = torch.empty(self.N, self.K // 2, dtype=torch.uint8, device=device)
        self.s_w = torch.empty(self.N, dtype=torch.float32, device=device)
        abi.sgat_prepare_weight(W, _dev(xf.inv_a_w, device=device), self.hb, self.Wq, self.s_w)
        del W
        self.We = None
        if e4m3_weights:
            self.We = torch.empty(self.N, self.K, dtype=torch.uint8, device=device)
            abi.w4_unpack_e4m3(self.Wq, self.We)
        self.workspace = torch.empty(abi.sgat_linear_workspace_size(self.L, self.K, self.tac is not None),
                                     dtype=torch.uint8, device=device)

    def run(self, X, mask, Y, stream=None):
        abi.sgat_linear(X, mask, self.a_m, self.a_u, self.hb, self.d_sh, self.d_m, self.d_u,
                        self.Wq, self.s_w, Y, self.workspace, bias=self.bias, tac_M=self.tac_M,
                        tac_d=self.tac_d, tac_g=self.tac_g, We=self.We, tac_Mp=self.tac_Mp, stream=stream)

    def buffers(self):
        """The layer's own code buffers (s_a and the E4M3 codes Xe; the packed
        codes are not needed, as the GEMM reads Xe) and TAC scratch, for
        launches that group several layers' quantisations or GEMMs."""
        if not hasattr(self, "Xe"):
            dev = self.s_w.device
            self.s_a = torch.empty(self.L, dtype=torch.float32, device=dev)
            self.Xe = torch.empty(self.L, self.K, dtype=torch.uint8, device=dev)
            self.tac_scratch = (torch.empty(self.L, self.K, dtype=self.dtype, device=dev)
                                if self.tac is not None else None)

    def quantize(self, X, mask, stream=None):
        """TAC (when the layer has it) and the state-guided quantisation of X
        into the layer's own code buffers (Xq, s_a, Xe), without the GEMM:
        for a grouped launch of several layers' GEMMs."""
        self.buffers()
        abi.sgat_quantize_act(X, mask, self.a_m, self.a_u, self.hb, self.d_sh, self.d_m, self.d_u, None,
                              self.s_a, Xe=self.Xe, stream=stream, tac_M=self.tac_M, tac_d=self.tac_d,
                              tac_g=self.tac_g, tac_Mp=self.tac_Mp, tac_scratch=self.tac_scratch)

    def int_ops(self, L=None):
        return 2 * (L or self.L) * self.N * self.K


class AttentionProjections:
    """QKV projection of X and TAC + O projection of Z for one step.

    qkv_pair_limit caps the CTA pairs of the QKV GEMM so that the O branch's
    TAC and quantiser can run beside it on the remaining SMs (0 = no cap,
    the default). On GB300 with the LLaDA shapes a cap of 48 pairs gave
    either 67-69 us or 82 us per replay, depending on which branch's CTAs
    the hardware placed first (against a steady 71-73 us uncapped), so it
    is off by default. Results do not depend on it."""

    def __init__(self, qkv_case, o_case, device="cuda", e4m3_weights=True, qkv_pair_limit=0, grouped=False):
        self.qkv = SgatLinear(qkv_case, device, e4m3_weights=e4m3_weights)
        self.o = SgatLinear(o_case, device, e4m3_weights=e4m3_weights)
        self.L = qkv_case.L
        self.X = _dev(qkv_case.X, self.qkv.dtype, device)
        self.Z = _dev(o_case.X, self.o.dtype, device)
        self.mask = _dev(qkv_case.mask, device=device)
        self.Y_qkv = torch.empty(self.L, self.qkv.N, dtype=self.qkv.out_dtype, device=device)
        self.Y_o = torch.empty(self.L, self.o.N, dtype=self.o.out_dtype, device=device)
        self.side = torch.cuda.Stream(device=device)
        self.qkv_pair_limit = qkv_pair_limit
        self.grouped = grouped if e4m3_weights else False
        self.KERNELS_PER_STEP = 3 if self.grouped is True else 4 if self.grouped else 5
        self.graph = None

    def step(self, stream=None):
        """The two projections are independent, so the O chain (TAC,
        quantiser, GEMM) runs on a side stream forked from `stream` and
        joined back at the end: its CUDA-core kernels overlap the QKV
        quantiser and the gaps between launches. The O chain is issued
        first, so that TAC starts beside the QKV quantiser. Outputs are
        identical to running the two projections one after the other.

        grouped=True: TAC on Z, then both quantisations in one launch
        (sgat_quantize_act_grouped) and both GEMMs in one launch
        (w4a4_gemm_grouped, the O tiles after the QKV tiles): three kernels
        on one stream. grouped="gemm": the O chain's TAC and quantiser run
        on the side stream beside the QKV quantiser, then the grouped GEMM."""
        main = stream if stream is not None else torch.cuda.current_stream()
        if self.grouped is True:
            q, o = self.qkv, self.o
            for lin in (q, o):
                lin.buffers()
            abi.tac_apply(self.Z, o.tac_M, o.tac_d, o.tac_g, o.tac_scratch, Mp=o.tac_Mp, stream=main)
            io = lambda lin, X: dict(X=X, mask=self.mask, a_m=lin.a_m, a_u=lin.a_u, d_sh=lin.d_sh, d_m=lin.d_m,
                                     d_u=lin.d_u, Xq=None, s_a=lin.s_a, Xe=lin.Xe)
            # the QKV rows do not depend on the TAC launch just before them
            abi.sgat_quantize_act_grouped(dict(io(q, self.X), independent=True), io(o, o.tac_scratch), q.hb,
                                          stream=main)
            abi.w4a4_gemm_grouped(q.Xe, q.s_a, q.We, q.s_w, self.Y_qkv, o.Xe, o.s_a, o.We, o.s_w, self.Y_o,
                                  bias0=q.bias, bias1=o.bias, weights_ready=True, stream=main)
            return
        if self.grouped:
            self.side.wait_stream(main)
            with torch.cuda.stream(self.side):
                self.o.quantize(self.Z, self.mask, self.side)
            self.qkv.quantize(self.X, self.mask, main)
            main.wait_stream(self.side)
            q, o = self.qkv, self.o
            abi.w4a4_gemm_grouped(q.Xe, q.s_a, q.We, q.s_w, self.Y_qkv, o.Xe, o.s_a, o.We, o.s_w, self.Y_o,
                                  bias0=q.bias, bias1=o.bias, stream=main)
            return
        self.side.wait_stream(main)
        with torch.cuda.stream(self.side):
            self.o.run(self.Z, self.mask, self.Y_o, self.side)
        prev = abi.set_gemm_pair_limit(self.qkv_pair_limit)
        try:
            self.qkv.run(self.X, self.mask, self.Y_qkv, main)
        finally:
            abi.set_gemm_pair_limit(prev)
        main.wait_stream(self.side)

    def capture(self):
        """Record one step in a CUDA graph (call after a warm-up step)."""
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self.step()
        torch.cuda.current_stream().wait_stream(s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.step()
        self.graph = g
        return g

    def replay(self):
        self.graph.replay()

    def int_ops(self):
        return self.qkv.int_ops() + self.o.int_ops()

    KERNELS_PER_STEP = 5   # quant + GEMM (QKV); TAC + quant + GEMM (O); 4 when grouped (one GEMM launch)
