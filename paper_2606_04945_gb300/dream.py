"""One Dream-7B-shaped (Qwen2.5-7B) transformer block, W4A4 with SGAT and
TAC, on the C ABI.

Per block (hidden 3584, 28 query heads over 4 key/value heads of 128, FFN
18944, bf16, 4 sequences of 2048 tokens):

    a  = RMSNorm(x) w1                                  glue_add_rmsnorm
    qkv = SGAT-W4A4(a) + b                               sgat_linear (Sec. 3.2)
    q, k = RoPE(q, k)                                    glue_rope
    z  = TAC(Q8(softmax(q k^T / sqrt 128)) Q4(v))        attention_pv_tac_gqa,
                                                         per sequence (Sec. 3.3)
    x1 = x + SGAT-W4A4(z)                                sgat_linear (O)
    a2 = RMSNorm(x1) w2                                  glue_add_rmsnorm (fused add)
    g  = silu(gate) up of SGAT-W4A4(a2)                  sgat_linear_swiglu
    x2 = x1 + SGAT-W4A4(g)                               sgat_linear (down), glue_add_rmsnorm

Every step runs in libstarq kernels; torch only holds the buffers. The mask
bit of each token selects its transform in every quantised linear. TAC is
applied in the attention kernel's epilogue, so the O projection's
sgat_linear takes no TAC of its own.
"""

import numpy as np
import torch

from . import abi

BF16 = torch.bfloat16


def _dev(x, dtype=None, device="cuda"):
    t = torch.from_numpy(np.ascontiguousarray(x))
    return (t.to(dtype) if dtype is not None else t).to(device)


class _Linear:
    """A quantised linear of the block: folded int4 weight (Eq. 12), its E4M3
    copy, per-channel scales, the two state transforms and a workspace."""

    def __init__(self, W, xf, L, bias=None, swiglu=False, device="cuda"):
        self.N, self.K = W.shape
        self.xf = xf
        self.swiglu = swiglu
        self.a_m, self.a_u = _dev(xf.a_m, device=device), _dev(xf.a_u, device=device)
        self.bias = _dev(bias, device=device) if bias is not None else None
        W16 = _dev(W, BF16, device)
        if swiglu:                        # gate rows 0..F-1, up rows F..2F-1 -> interleaved by 16
            W16 = W16[abi.swiglu_row_order(self.N // 2, device)].contiguous()
        self.Wq = torch.empty(self.N, self.K // 2, dtype=torch.uint8, device=device)
        self.s_w = torch.empty(self.N, dtype=torch.float32, device=device)
        abi.sgat_prepare_weight(W16, _dev(xf.inv_a_w, device=device), xf.hb, self.Wq, self.s_w)
        del W16
        self.We = torch.empty(self.N, self.K, dtype=torch.uint8, device=device)
        abi.w4_unpack_e4m3(self.Wq, self.We)
        self.workspace = torch.empty(abi.sgat_linear_workspace_size(L, self.K, False), dtype=torch.uint8,
                                     device=device)

    def run(self, X, mask, Y, stream=None):
        xf = self.xf
        fn = abi.sgat_linear_swiglu if self.swiglu else abi.sgat_linear
        fn(X, mask, self.a_m, self.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, self.Wq, self.s_w, Y, self.workspace,
           bias=self.bias, We=self.We, stream=stream)

    def int_ops(self, L):
        return 2 * L * self.N * self.K


class DreamBlock:
    KERNELS = ("glue_add_rmsnorm", "sgat_linear (QKV)", "glue_rope", "attention_pv_tac_gqa x batch",
               "sgat_linear (O)", "glue_add_rmsnorm", "sgat_linear_swiglu", "sgat_linear (down)",
               "glue_add_rmsnorm")

    def __init__(self, case, device="cuda"):
        c = case
        self.case = c
        self.L, self.H, self.F = c.L, c.hidden, c.ffn
        self.heads, self.kv_heads = c.heads, c.kv_heads
        L, H, F = self.L, self.H, self.F
        self.qkv = _Linear(c.W_qkv, c.xf_qkv, L, bias=c.b_qkv, device=device)
        self.o = _Linear(c.W_o, c.xf_o, L, device=device)
        self.gu = _Linear(np.concatenate([c.W_gate, c.W_up]), c.xf_gu, L, swiglu=True, device=device)
        self.down = _Linear(c.W_down, c.xf_down, L, device=device)
        self.w_ln1, self.w_ln2 = _dev(c.w_ln1, device=device), _dev(c.w_ln2, device=device)
        self.tac_M, self.tac_d = _dev(c.tac.M, device=device), _dev(c.tac.d, device=device)
        self.tac_Mp = torch.empty(abi.tac_prepared_bytes(H, 128), dtype=torch.uint8, device=device)
        abi.tac_prepare(self.tac_M, 128, torch.float16, self.tac_Mp)      # the attention's TAC runs on fp16 halves
        self.X = _dev(c.X, BF16, device)
        self.mask = _dev(c.mask, device=device)
        self.pos = _dev(c.pos.astype(np.int32), device=device)
        t = lambda *s: torch.empty(*s, dtype=BF16, device=device)
        nqkv = (self.heads + 2 * self.kv_heads) * 128
        self.buf = dict(a=t(L, H), qkv=t(L, nqkv), z=t(L, H), o=t(L, H), x1=t(L, H), a2=t(L, H),
                        g=t(L, F), d=t(L, H), out=t(L, H))
        self.attn_ws = torch.empty(abi.attention_pv_tac_workspace_size(c.seq, self.kv_heads), dtype=torch.uint8,
                                   device=device)
        self.graph = None

    def attention(self, qkv, z, stream=None):
        c = self.case
        Cq, Ckv = self.heads * 128, self.kv_heads * 128
        for b in range(c.batch):
            rows = slice(b * c.seq, (b + 1) * c.seq)
            q = qkv[rows, :Cq]
            k = qkv[rows, Cq:Cq + Ckv]
            v = qkv[rows, Cq + Ckv:]
            abi.attention_pv_tac(q, k, v, self.heads, self.tac_Mp, self.tac_d, z[rows], workspace=self.attn_ws,
                                 Hkv=self.kv_heads, stream=stream)

    def forward(self, hook=None, stream=None):
        """One pass of the block over self.X; returns the output buffer.
        hook(name, tensor) sees every intermediate (for tests)."""
        c, b = self.case, self.buf
        hk = hook or (lambda name, t: None)
        abi.add_rmsnorm(self.X, self.w_ln1, b["a"], eps=c.eps, stream=stream)
        hk("a", b["a"])
        self.qkv.run(b["a"], self.mask, b["qkv"], stream)
        if hook is not None:
            hook("qkv", b["qkv"].clone())
        abi.rope(b["qkv"], self.heads + self.kv_heads, self.pos, c.rope_theta, stream=stream)
        hk("qkv_rope", b["qkv"])
        self.attention(b["qkv"], b["z"], stream)
        hk("z", b["z"])
        self.o.run(b["z"], self.mask, b["o"], stream)
        hk("o", b["o"])
        abi.add_rmsnorm(b["o"], self.w_ln2, b["a2"], R=self.X, h_out=b["x1"], eps=c.eps, stream=stream)
        hk("x1", b["x1"])
        hk("a2", b["a2"])
        self.gu.run(b["a2"], self.mask, b["g"], stream)
        hk("g", b["g"])
        self.down.run(b["g"], self.mask, b["d"], stream)
        hk("d", b["d"])
        abi.add_rmsnorm(b["d"], None, None, R=b["x1"], h_out=b["out"], stream=stream)
        return b["out"]

    def capture(self):
        """Record one block pass in a CUDA graph (after an eager pass)."""
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self.forward()
        torch.cuda.current_stream().wait_stream(s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.forward()
        self.graph = g
        return g

    def replay(self):
        self.graph.replay()

    def int_ops(self):
        L = self.L
        return self.qkv.int_ops(L) + self.o.int_ops(L) + self.gu.int_ops(L) + self.down.int_ops(L)

    def kernel_launches(self):
        """Kernels of one pass: three norms, rope, 4 x (V quantiser +
        attention), and quantiser + GEMM for each of the four linears."""
        return 3 + 1 + 2 * self.case.batch + 4 * 2
