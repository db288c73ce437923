"""Iterative denoising with a LLaDA-8B-shaped stack of SGAT W4A4 layers.

A stack of pre-norm transformer blocks (hidden 4096, FFN 12288, 32 heads of
128, bidirectional attention), random-init weights, run over the denoising
trajectory of one sequence: 1024 positions, the last 256 generated; they
start masked and 4 are unmasked per step (seeded random confidence), each
with a seeded random token, so the trajectory does not depend on the
outputs. Per block:

    h = RMSNorm(x)
    q, k, v = SGAT-W4A4(h)                  QKV 4096 -> 12288 (Sec. 3.2)
    a = softmax(RoPE(q) RoPE(k)^T / sqrt(128)) v          (bidirectional)
    x = x + SGAT-W4A4(TAC(a))               O 4096 -> 4096, TAC 128 x 128 per head (Sec. 3.3)
    h = RMSNorm(x)
    g, u = SGAT-W4A4(h)                     gate+up 4096 -> 2 x 12288
    x = x + SGAT-W4A4(silu(g) u)            down 12288 -> 4096

Every linear is one `sgat_linear` call of the C ABI with the token's mask
bit selecting its transform; the gate+up projection is `sgat_linear_swiglu`,
which applies silu(g) u in the GEMM epilogue. RMSNorm, RoPE, attention and
the residuals are glue (torch ops on the GPU), not part of the quantised
path; the 16-bit baseline applies SwiGLU as glue too.
The same stack with 16-bit GEMMs (`fp16_gemm_ref`, no quantisation, no
TAC) is the unquantised baseline for the per-step output drift.

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


def rms_norm(x, eps=1e-6):
    xf = x.float()
    return (xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + eps)).to(x.dtype)


def rope_tables(L, d, device, base=10000.0):
    inv = 1.0 / (base ** (torch.arange(0, d, 2, device=device, dtype=torch.float32) / d))
    ang = torch.arange(L, device=device, dtype=torch.float32)[:, None] * inv[None]
    return torch.cos(ang), torch.sin(ang)


def apply_rope(t, cos, sin):
    # t [heads, L, d]; rotate the two halves of each head
    d2 = t.shape[-1] // 2
    t1, t2 = t[..., :d2].float(), t[..., d2:].float()
    return torch.cat([t1 * cos - t2 * sin, t1 * sin + t2 * cos], -1).to(t.dtype)


class QLinear:
    """One linear of the stack: the 16-bit weight (baseline), its prepared
    W4A4 form (packed int4 codes, E4M3 copy, per-channel scales), the SGAT
    transforms, optional TAC, and a workspace."""

    def __init__(self, W16, L, tac=None, swiglu=False):
        self.W16 = W16
        self.N, self.K = W16.shape
        self.L = L
        self.tac = tac
        # gate+up of the MLP: the W4A4 form keeps the rows in
        # swiglu_row_order and writes silu(gate) * up [L][N / 2]
        self.swiglu = swiglu
        self.sgat = None
        self.tac_M = self.tac_d = self.tac_Mp = None
        if tac is not None:
            dev = W16.device
            self.tac_M = torch.from_numpy(tac.M).to(dev)
            self.tac_d = torch.from_numpy(tac.d).to(dev)
            self.tac_Mp = torch.empty(abi.tac_prepared_bytes(self.K, tac.g), dtype=torch.uint8, device=dev)
            abi.tac_prepare(self.tac_M, tac.g, W16.dtype, self.tac_Mp)

    def tac_out(self, X):
        """TAC of the linear's input (float32), as sgat_linear applies it."""
        Z = torch.empty(X.shape, dtype=torch.float32, device=X.device)
        abi.tac_apply(X, self.tac_M, self.tac_d, self.tac.g, Z, Mp=self.tac_Mp)
        return Z

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
                        self.workspace, tac_M=self.tac_M, tac_d=self.tac_d,
                        tac_g=self.tac.g if self.tac is not None else 0, We=self.We, tac_Mp=self.tac_Mp)

    def fp16(self, X, Y):
        abi.fp16_gemm_ref(X, self.W16, Y)


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
                o=QLinear(w(c.hidden, c.hidden), c.seq, tac=inputs.make_tac(rng, c.hidden, c.tac_block)),
                gu=QLinear(w(2 * c.ffn, c.hidden), c.seq, swiglu=True),
                down=QLinear(w(c.hidden, c.ffn), c.seq)))
        self.cos, self.sin = rope_tables(c.seq, c.hidden // c.heads, device)
        # denoising trajectory: prompt tokens, then masked positions unmasked
        # four per step in a seeded order with seeded tokens
        self.prompt = torch.from_numpy(rng.integers(1, c.vocab, c.seq - c.gen)).to(device)
        self.order = rng.permutation(c.gen)
        self.new_tokens = rng.integers(1, c.vocab, c.gen)
        L, H, F = c.seq, c.hidden, c.ffn
        t = lambda *s: torch.empty(*s, dtype=torch.float16, device=device)
        self.buf = dict(qkv=t(L, 3 * H), attn=t(L, H), o=t(L, H), gu=t(L, 2 * F), act=t(L, F), down=t(L, H))

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
    def _attention(self, qkv):
        c = self.cfg
        L, H, nh = c.seq, c.hidden, c.heads
        d = H // nh
        q, k, v = qkv.view(L, 3, nh, d).permute(1, 2, 0, 3)          # [3][heads][L][d]
        q, k = apply_rope(q, self.cos, self.sin), apply_rope(k, self.cos, self.sin)
        a = torch.nn.functional.scaled_dot_product_attention(q[None], k[None], v[None])[0]
        return a.permute(1, 0, 2).reshape(L, H).contiguous()

    def forward(self, tok, mask, quantised=True, hook=None):
        """One denoising step of the whole stack; returns the final hidden
        state. tok: token ids (device, long), mask: mask bits (numpy or
        device uint8). `hook(layer, name, linear, X, Y)` runs after each
        quantised linear (X its input, Y its output) for inspection."""
        mask_d = mask if torch.is_tensor(mask) else torch.from_numpy(mask).to(self.device)
        return self._forward(tok, mask_d, quantised, hook)

    def _forward(self, tok, mask_d, quantised, hook):
        c = self.cfg
        b = self.buf
        x = self.embed[tok].clone()
        for li, blk in enumerate(self.blocks):
            h = rms_norm(x)
            self._lin(blk["qkv"], h, mask_d, b["qkv"], quantised, hook, li, "qkv")
            a = self._attention(b["qkv"])
            b["attn"].copy_(a)
            self._lin(blk["o"], b["attn"], mask_d, b["o"], quantised, hook, li, "o")
            x = x + b["o"]
            h = rms_norm(x)
            if quantised:                                 # silu(gate) * up in the GEMM epilogue
                self._lin(blk["gu"], h, mask_d, b["act"], True, hook, li, "gu")
            else:
                blk["gu"].fp16(h, b["gu"])
                gt, up = b["gu"][:, : c.ffn], b["gu"][:, c.ffn:]
                b["act"].copy_((torch.nn.functional.silu(gt.float()) * up.float()).half())
            self._lin(blk["down"], b["act"], mask_d, b["down"], quantised, hook, li, "down")
            x = x + b["down"]
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
        """Per-linear smoothing from a 16-bit pass over the initial state."""
        tok, mask = self.state(0)
        c = self.cfg
        b = self.buf
        x = self.embed[tok].clone()
        for blk in self.blocks:
            h = rms_norm(x)
            blk["qkv"].fp16(h, b["qkv"])
            blk["qkv"].calibrate(h, mask)
            b["attn"].copy_(self._attention(b["qkv"]))
            blk["o"].calibrate(blk["o"].tac_out(b["attn"]), mask)   # its quantiser sees TAC(a)
            blk["o"].fp16(b["attn"], b["o"])
            x = x + b["o"]
            h = rms_norm(x)
            blk["gu"].calibrate(h, mask)
            blk["gu"].fp16(h, b["gu"])
            gt, up = b["gu"][:, : c.ffn], b["gu"][:, c.ffn:]
            b["act"].copy_((torch.nn.functional.silu(gt.float()) * up.float()).half())
            blk["down"].calibrate(b["act"], mask)
            blk["down"].fp16(b["act"], b["down"])
            x = x + b["down"]

    def linear_int_ops(self):
        c = self.cfg
        per_layer = 2 * c.seq * (3 * c.hidden * c.hidden + c.hidden * c.hidden + 2 * c.ffn * c.hidden
                                 + c.hidden * c.ffn)
        return c.layers * per_layer
