"""Iterative denoising with a LLaDA-8B-shaped stack of SGAT W4A4 layers.

A stack of pre-norm transformer blocks (hidden 4096, FFN 12288, 32 heads of
128, bidirectional attention), random-init weights, run over the denoising
trajectory of one sequence: 1024 positions, the last 256 generated; they
start masked and 4 are unmasked per step (seeded random confidence), each
with a seeded random token, so the trajectory does not depend on the
outputs. Per block:

    h = RMSNorm(x)                          glue_add_rmsnorm
    q, k, v = SGAT-W4A4(h)                  QKV 4096 -> 12288 (Sec. 3.2)
    q, k = RoPE(q, k)                       glue_rope
    a = TAC(Q8(softmax(q k^T / sqrt(128))) Q4(v))     attention_pv_tac: the
                                            quantised softmax-value product with
                                            TAC, 128 x 128 per head (Sec. 3.3)
    x = x + SGAT-W4A4(a); h = RMSNorm(x)    O 4096 -> 4096; glue_add_rmsnorm
    g, u = SGAT-W4A4(h)                     gate+up 4096 -> 2 x 12288
    x = x + SGAT-W4A4(silu(g) u)            down 12288 -> 4096

Every step runs in libstarq kernels: every linear is one `sgat_linear` call
with the token's mask bit selecting its transform (the gate+up projection
is `sgat_linear_swiglu`, with silu(g) u in the GEMM epilogue), attention is
the quantised product whose output TAC compensates, and RMSNorm, RoPE and
the residuals are the library's glue kernels.
The same stack with 16-bit GEMMs (`fp16_gemm_ref`), unquantised attention
(torch's fp16 SDPA) and no TAC is the unquantised baseline for the
per-step output drift; it applies SwiGLU as glue.

The per-state smoothing of every linear is calibrated on that linear's
input in one 16-bit pass over the initial state (synthetic calibration).
"""

from dataclasses import dataclass

import numpy as np
import torch

from . import abi, inputs


@dataclass
class StackConfig:
    hidden: int = 4096
    ffn: int = 12288
    heads: int = 32
    layers: int = 4
    seq: int = 1024
    gen: int = 256
    steps: int = 64
    unmask_per_step: int = 4
    vocab: int = 8192
    tac_block: int = 128
    seed: int = 0


ROPE_THETA = 10000.0
EPS = 1e-6


class QLinear:
    """One linear of the stack: the 16-bit weight (baseline), its prepared
    W4A4 form (packed int4 codes, E4M3 copy, per-channel scales), the SGAT
    transforms, optional TAC, and a workspace."""

    def __init__(self, W16, L, swiglu=False):
        self.W16 = W16
        self.N, self.K = W16.shape
        self.L = L
        self.tac = None
        # gate+up of the MLP: the W4A4 form keeps the rows in
        # swiglu_row_order and writes silu(gate) * up [L][N / 2]
        self.swiglu = swiglu
        self.sgat = None

    def calibrate(self, X, mask):
        xf = inputs.make_sgat(X.float().cpu().numpy(), mask)
        dev = self.W16.device
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        self.sgat = xf
        self.a_m, self.a_u = t(xf.a_m), t(xf.a_u)
        self.Wq = torch.empty(self.N, self.K // 2, dtype=torch.uint8, device=dev)
        self.s_w = torch.empty(self.N, dtype=torch.float32, device=dev)
        W = self.W16[abi.swiglu_row_order(self.N // 2, dev)] if self.swiglu else self.W16
        abi.sgat_prepare_weight(W, t(xf.inv_a_w), xf.hb, self.Wq, self.s_w)
        self.We = torch.empty(self.N, self.K, dtype=torch.uint8, device=dev)
        abi.w4_unpack_e4m3(self.Wq, self.We)
        self.workspace = torch.empty(abi.sgat_linear_workspace_size(self.L, self.K, self.tac is not None),
                                     dtype=torch.uint8, device=dev)

    def w4a4(self, X, mask, Y):
        xf = self.sgat
        if self.swiglu:
            abi.sgat_linear_swiglu(X, mask, self.a_m, self.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, self.Wq, self.s_w,
                                   Y, self.workspace, We=self.We)
            return
        abi.sgat_linear(X, mask, self.a_m, self.a_u, xf.hb, xf.d_sh, xf.d_m, xf.d_u, self.Wq, self.s_w, Y,
                        self.workspace, We=self.We)

    def fp16(self, X, Y):
        abi.fp16_gemm_ref(X, self.W16, Y)


class QAttention:
    """The quantised softmax-value product of one block with TAC in its
    epilogue (per-head 128 x 128 blocks, prepared once)."""

    def __init__(self, tac, L, heads, device):
        self.tac = tac
        self.heads = heads
        self.M = torch.from_numpy(tac.M).to(device)
        self.d = torch.from_numpy(tac.d).to(device)
        self.Mp = torch.empty(abi.tac_prepared_bytes(tac.C, tac.g), dtype=torch.uint8, device=device)
        abi.tac_prepare(self.M, tac.g, torch.float16, self.Mp)
        self.workspace = torch.empty(abi.attention_pv_tac_workspace_size(L, heads), dtype=torch.uint8, device=device)

    def run(self, qkv, out, **dbg):
        C = self.heads * 128
        abi.attention_pv_tac(qkv[:, :C], qkv[:, C:2 * C], qkv[:, 2 * C:], self.heads, self.Mp, self.d, out,
                             workspace=self.workspace, **dbg)

    def tac_f32(self, A):
        """TAC of a 16-bit attention output, in float32 (calibration)."""
        Z = torch.empty(A.shape, dtype=torch.float32, device=A.device)
        abi.tac_apply(A, self.M, self.d, self.tac.g, Z, Mp=self.Mp)
        return Z


class DenoiseStack:
    def __init__(self, cfg: StackConfig, device="cuda"):
        self.cfg = cfg
        c = cfg
        self.device = device
        g = torch.Generator(device=device).manual_seed(c.seed)
        rng = np.random.default_rng(c.seed)
        w = lambda n, k: (torch.randn(n, k, generator=g, device=device) * 0.02).half()
        self.embed = torch.randn(c.vocab, c.hidden, generator=g, device=device).half()
        self.mask_id = 0
        self.blocks = []
        for _ in range(c.layers):
            self.blocks.append(dict(
                qkv=QLinear(w(3 * c.hidden, c.hidden), c.seq),
                attn=QAttention(inputs.make_tac(rng, c.hidden, c.tac_block), c.seq, c.heads, device),
                o=QLinear(w(c.hidden, c.hidden), c.seq),
                gu=QLinear(w(2 * c.ffn, c.hidden), c.seq, swiglu=True),
                down=QLinear(w(c.hidden, c.ffn), c.seq)))
        self.ones = torch.ones(c.hidden, dtype=torch.float32, device=device)
        self.pos = torch.arange(c.seq, dtype=torch.int32, device=device)
        # denoising trajectory: prompt tokens, then masked positions unmasked
        # four per step in a seeded order with seeded tokens
        self.prompt = torch.from_numpy(rng.integers(1, c.vocab, c.seq - c.gen)).to(device)
        self.order = rng.permutation(c.gen)
        self.new_tokens = rng.integers(1, c.vocab, c.gen)
        L, H, F = c.seq, c.hidden, c.ffn
        t = lambda *s: torch.empty(*s, dtype=torch.float16, device=device)
        self.buf = dict(x=t(L, H), h=t(L, H), qkv=t(L, 3 * H), attn=t(L, H), o=t(L, H), gu=t(L, 2 * F),
                        act=t(L, F), down=t(L, H))

    # -- trajectory -----------------------------------------------------
    def state(self, step):
        """Token ids and mask bits (1 = masked) seen by denoising step `step`."""
        c = self.cfg
        tok = torch.full((c.seq,), self.mask_id, dtype=torch.long, device=self.device)
        tok[: c.seq - c.gen] = self.prompt
        mask = np.zeros(c.seq, np.uint8)
        mask[c.seq - c.gen:] = 1
        done = self.order[: step * c.unmask_per_step]
        pos = c.seq - c.gen + done
        tok[torch.from_numpy(pos).to(self.device)] = torch.from_numpy(self.new_tokens[done]).to(self.device)
        mask[pos] = 0
        return tok, mask

    # -- one forward pass ------------------------------------------------
    def _sdpa(self, qkv):
        """Unquantised attention of the 16-bit baseline (on roped q, k)."""
        c = self.cfg
        L, H, nh = c.seq, c.hidden, c.heads
        q, k, v = qkv.view(L, 3, nh, H // nh).permute(1, 2, 0, 3)          # [3][heads][L][d]
        a = torch.nn.functional.scaled_dot_product_attention(q[None], k[None], v[None])[0]
        return a.permute(1, 0, 2).reshape(L, H)

    def forward(self, tok, mask, quantised=True, hook=None):
        """One denoising step of the whole stack; returns the final hidden
        state. tok: token ids (device, long), mask: mask bits (numpy or
        device uint8). `hook(layer, name, module, X, Y)` runs after each
        quantised linear (X its input, Y its output) and after the quantised
        attention (X the roped QKV output, Y the TAC-compensated output)."""
        mask_d = mask if torch.is_tensor(mask) else torch.from_numpy(mask).to(self.device)
        return self._forward(tok, mask_d, quantised, hook)

    def _forward(self, tok, mask_d, quantised, hook):
        c = self.cfg
        b = self.buf
        H, nh = c.hidden, c.heads
        x, h = b["x"], b["h"]
        x.copy_(self.embed[tok])
        abi.add_rmsnorm(x, self.ones, h, eps=EPS)
        for li, blk in enumerate(self.blocks):
            self._lin(blk["qkv"], h, mask_d, b["qkv"], quantised, hook, li, "qkv")
            abi.rope(b["qkv"], 2 * nh, self.pos, ROPE_THETA)
            if quantised:
                blk["attn"].run(b["qkv"], b["attn"])
                if hook is not None:
                    hook(li, "attn", blk["attn"], b["qkv"], b["attn"])
            else:
                b["attn"].copy_(self._sdpa(b["qkv"]))
            self._lin(blk["o"], b["attn"], mask_d, b["o"], quantised, hook, li, "o")
            abi.add_rmsnorm(b["o"], self.ones, h, R=x, h_out=x, eps=EPS)        # x += o; h = norm(x)
            if quantised:                                 # silu(gate) * up in the GEMM epilogue
                self._lin(blk["gu"], h, mask_d, b["act"], True, hook, li, "gu")
            else:
                blk["gu"].fp16(h, b["gu"])
                gt, up = b["gu"][:, : c.ffn], b["gu"][:, c.ffn:]
                b["act"].copy_((torch.nn.functional.silu(gt.float()) * up.float()).half())
            self._lin(blk["down"], b["act"], mask_d, b["down"], quantised, hook, li, "down")
            last = li == len(self.blocks) - 1
            # x += down; h = norm(x) for the next block
            abi.add_rmsnorm(b["down"], self.ones, None if last else h, R=x, h_out=x, eps=EPS)
        return x

    def capture(self, quantised=True):
        """Record one step in a CUDA graph over static token / mask buffers;
        returns (graph, tok buffer, mask buffer, output). Fill the buffers
        (set_state) and replay for each step."""
        c = self.cfg
        tok_s = torch.zeros(c.seq, dtype=torch.long, device=self.device)
        mask_s = torch.zeros(c.seq, dtype=torch.uint8, device=self.device)
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            self._forward(tok_s, mask_s, quantised, None)
        torch.cuda.current_stream().wait_stream(side)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            out = self._forward(tok_s, mask_s, quantised, None)
        return g, tok_s, mask_s, out

    def set_state(self, step, tok_s, mask_s):
        tok, mask = self.state(step)
        tok_s.copy_(tok)
        mask_s.copy_(torch.from_numpy(mask))

    @staticmethod
    def _lin(lin, X, mask_d, Y, quantised, hook, li, name):
        if quantised:
            lin.w4a4(X, mask_d, Y)
            if hook is not None:
                hook(li, name, lin, X, Y)
        else:
            lin.fp16(X, Y)

    def calibrate(self):
        """Per-linear smoothing from a 16-bit pass over the initial state
        (the O projection's on the TAC of the unquantised attention)."""
        tok, mask = self.state(0)
        c = self.cfg
        b = self.buf
        x, h = b["x"], b["h"]
        x.copy_(self.embed[tok])
        abi.add_rmsnorm(x, self.ones, h, eps=EPS)
        for blk in self.blocks:
            blk["qkv"].fp16(h, b["qkv"])
            blk["qkv"].calibrate(h, mask)
            abi.rope(b["qkv"], 2 * c.heads, self.pos, ROPE_THETA)
            b["attn"].copy_(self._sdpa(b["qkv"]))
            blk["o"].calibrate(blk["attn"].tac_f32(b["attn"]), mask)
            blk["o"].fp16(b["attn"], b["o"])
            abi.add_rmsnorm(b["o"], self.ones, h, R=x, h_out=x, eps=EPS)
            blk["gu"].calibrate(h, mask)
            blk["gu"].fp16(h, b["gu"])
            gt, up = b["gu"][:, : c.ffn], b["gu"][:, c.ffn:]
            b["act"].copy_((torch.nn.functional.silu(gt.float()) * up.float()).half())
            blk["down"].calibrate(b["act"], mask)
            blk["down"].fp16(b["act"], b["down"])
            abi.add_rmsnorm(b["down"], self.ones, h, R=x, h_out=x, eps=EPS)

    def linear_int_ops(self):
        c = self.cfg
        per_layer = 2 * c.seq * (3 * c.hidden * c.hidden + c.hidden * c.hidden + 2 * c.ffn * c.hidden
                                 + c.hidden * c.ffn)
        return c.layers * per_layer
