"""Oracle: the glue of a transformer block around its quantised linears,
float64. Test infrastructure only (see the package docstring): the CUDA
path never imports this module.

These ops are not the paper's method (Sec. 3 quantises the linears and the
softmax-value product); the quantised Dream-7B / LLaDA-8B blocks run them
between the projections (residual stream, pre-norm RMSNorm, rotary
position embedding, the SwiGLU MLP). The definitions are the standard ones
of the LLaMA / Qwen2 family:

* ``rmsnorm``: y = h / sqrt(mean(h^2) + eps) * w per row;
* ``rope``: per head of d channels and i < d / 2, the pair (x_i, x_{i+d/2})
  rotated by the angle pos * theta^(-2 i / d) (the rotate-half form);
* ``swiglu``: silu(gate) * up, silu(x) = x / (1 + exp(-x)).
"""

import numpy as np

F64 = np.float64


def rmsnorm(h, w, eps):
    """Row-wise RMSNorm of h [L][K] with gain w [K] (float64)."""
    h = np.asarray(h, F64)
    ms = np.mean(h * h, axis=1, keepdims=True)
    return h / np.sqrt(ms + eps) * np.asarray(w, F64)[None, :]


def rope_frequencies(theta, d=128):
    """f_i = theta^(-2 i / d) for i < d / 2."""
    i = np.arange(d // 2, dtype=F64)
    return theta ** (-2.0 * i / d)


def rope(x, pos, heads, theta, d=128, angles=None):
    """Rotate the first `heads` heads of d channels of every row of x [L][*]
    by the token positions pos [L]; columns past heads * d are returned
    unchanged. angles [L][d / 2] (optional) overrides pos * f_i, e.g. with
    the float32 angles a kernel forms."""
    x = np.array(x, dtype=F64)
    if angles is None:
        ang = np.asarray(pos, F64)[:, None] * rope_frequencies(theta, d)[None, :]
    else:
        ang = np.asarray(angles, F64)
    c, s = np.cos(ang), np.sin(ang)
    for h in range(heads):
        a = x[:, h * d:h * d + d // 2].copy()
        b = x[:, h * d + d // 2:(h + 1) * d].copy()
        x[:, h * d:h * d + d // 2] = a * c - b * s
        x[:, h * d + d // 2:(h + 1) * d] = b * c + a * s
    return x


def swiglu(gate, up):
    """silu(gate) * up (float64)."""
    g = np.asarray(gate, F64)
    return g / (1.0 + np.exp(-g)) * np.asarray(up, F64)
