"""CPU oracle for precomputing F with the f-gram model A_fgram.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import this module. The product path never
imports it and has no CPU fallback through it.

What it computes. Algorithm 1's training branch embeds an f-gram
w = (s_j .. s_i) as A_fgram(T(s_j), .., T(s_i)), the output of the model at
the f-gram's final token; at inference that vector is read from the table F,
so F(w) is A_fgram applied once to each f-gram's token embeddings and stored
(Sec. 3.2: F is precomputed after training; processing an f-gram is running
a short sequence of length |w| through a standard transformer). The model
replicates the baseline architecture without its token embedding layer
(Sec. 4.1), and Appendix F ("Implementation Details") gives its position
scheme: an absolute position embedding layer whose number of positions is the
longest n-gram length in V_fgram, with the f-grams of a batch padded to the
longest one in the batch. The architecture used here:

  x_0[j] = T(s_{j'}) + P[j],  j = 0..n-1 counted from the f-gram's first
           token (P: [max_pos x d] learned absolute position embeddings)
  per layer:  h = x + Attn(LN(x));  x = h + MLP(LN(h))
    LN(v)   = (v - mean(v)) / sqrt(var(v) + 1e-5)           (no scale or bias)
    Attn    = causal multi-head attention, q, k, v = LN(x) W_q^T, W_k^T, W_v^T,
              scores / sqrt(hd), softmax, heads concatenated, then W_o^T
    MLP     = (silu(LN(h) W_gate^T) * (LN(h) W_up^T)) W_down^T
  F(w) = LN(x_L) at the last position (the f-gram's last token).

Padding to the batch's longest f-gram sits after the last token and the
attention is causal, so the last token's output does not depend on it: each
f-gram is evaluated here on its own n positions.

A second position scheme, rotary embeddings on q and k instead of P
(rotate-half pairs (i, i + hd/2), angle pos * 10000^(-2i/hd), positions
0..n-1), is the option of models whose ``position`` is "rotary"; it is not
the paper's.

All arithmetic is float64 numpy. With ``emulate_bf16`` the values the GPU
stores as bf16 are rounded to bf16 (nearest, ties to even) at the same points:
the model input x_0, the residual stream after each addition, LN outputs,
q/k/v, the attention output, the MLP activation and F. Without it the forward
is exact float64. Weights come as the packed bf16 buffer that
``synth.model_weights_cpu`` describes.
"""

from __future__ import annotations

import numpy as np

LN_EPS = 1e-5
ROPE_BASE = 10000.0


def bf16_to_f64(u16: np.ndarray) -> np.ndarray:
    """Raw bf16 words -> float64 (exact)."""
    return (np.asarray(u16, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def bf16_round(x: np.ndarray) -> np.ndarray:
    """float64 -> nearest bf16 value (ties to even), returned as float64.

    bf16 keeps 8 significant bits: scale each value into [2^7, 2^8) by its
    binary exponent and round to an integer there (numpy rounds half to even).
    """
    x = np.asarray(x, np.float64)
    out = np.zeros_like(x)
    nz = x != 0
    m, e = np.frexp(x[nz])                 # x = m 2^e, 0.5 <= |m| < 1
    out[nz] = np.ldexp(np.round(m * 256.0), e - 8)
    return out


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """float64 values that are bf16-representable -> raw bf16 words."""
    return (np.asarray(x, np.float32).view(np.uint32) >> 16).astype(np.uint16)


class Weights:
    """Per-layer float64 matrices unpacked from the packed bf16 buffer, and
    the position table P for the absolute scheme."""

    def __init__(self, packed: np.ndarray, model):
        self.m = model
        self.position = model.position
        d, f = model.d, model.ffw
        self.layers = []
        for layer in range(model.n_layers):
            mats = {}
            for name, r, c in model.shapes():
                off = model.offset(layer, name)
                mats[name] = bf16_to_f64(packed[off:off + r * c]).reshape(r, c)
            gu = mats.pop("gu").reshape(f // 16, 2, 16, d)
            mats["gate"] = gu[:, 0].reshape(f, d)
            mats["up"] = gu[:, 1].reshape(f, d)
            qkv = mats.pop("qkv")
            mats["q"], mats["k"], mats["v"] = qkv[:d], qkv[d:2 * d], qkv[2 * d:]
            self.layers.append(mats)
        self.P = None
        if self.position == "absolute":
            off = model.pos_offset
            self.P = bf16_to_f64(packed[off:off + model.max_pos * d]).reshape(model.max_pos, d)
        elif self.position != "rotary":
            raise ValueError(f"unknown position scheme {self.position}")


def position_rows(W: Weights, n: int) -> np.ndarray:
    """What the position scheme adds to the n input rows: P[0..n-1] for
    absolute positions (position j is the j-th token of the f-gram), zero for
    rotary ones."""
    if W.position != "absolute":
        return np.zeros((n, W.m.d))
    if n > W.P.shape[0]:
        raise ValueError(f"f-gram of {n} tokens, but only {W.P.shape[0]} positions")
    return W.P[:n]


def layer_norm(x: np.ndarray) -> np.ndarray:
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + LN_EPS)


def rope(x: np.ndarray, pos: np.ndarray) -> np.ndarray:
    """Rotary embedding of x [n, hd] at positions pos [n] (rotate-half pairs)."""
    hd = x.shape[-1]
    half = hd // 2
    theta = ROPE_BASE ** (-2.0 * np.arange(half) / hd)          # [half]
    ang = pos[:, None].astype(np.float64) * theta[None, :]     # [n, half]
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[:, :half], x[:, half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def attention(q, k, v, n_heads, rotary: bool = False):
    """Causal multi-head attention; q, k, v [n, d]. With ``rotary`` the rotary
    embedding is applied to q and k first."""
    n, d = q.shape
    hd = d // n_heads
    pos = np.arange(n)
    out = np.empty((n, d))
    for h in range(n_heads):
        sl = slice(h * hd, (h + 1) * hd)
        qh, kh, vh = q[:, sl], k[:, sl], v[:, sl]
        if rotary:
            qh, kh = rope(qh, pos), rope(kh, pos)
        scores = qh @ kh.T / np.sqrt(hd)
        scores = np.where(np.tril(np.ones((n, n), bool)), scores, -np.inf)
        p = np.exp(scores - scores.max(axis=1, keepdims=True))
        p /= p.sum(axis=1, keepdims=True)
        out[:, sl] = p @ vh
    return out


def silu(x):
    return x / (1.0 + np.exp(-x))


def forward_states(x0: np.ndarray, W: Weights, emulate_bf16: bool = True):
    """Residual stream after the last layer, [n, d] (before the final LN);
    x0 is the model input (token rows plus position rows)."""
    r = bf16_round if emulate_bf16 else (lambda a: a)
    rotary = W.position == "rotary"
    x = r(np.asarray(x0, np.float64))
    for L in W.layers:
        xn = r(layer_norm(x))
        q, k, v = r(xn @ L["q"].T), r(xn @ L["k"].T), r(xn @ L["v"].T)
        o = r(attention(q, k, v, W.m.n_heads, rotary))
        x = r(x + o @ L["o"].T)
        xn = r(layer_norm(x))
        a = r(silu(xn @ L["gate"].T) * (xn @ L["up"].T))
        x = r(x + a @ L["down"].T)
    return x


def model_input(tokens, T_rows: np.ndarray, W: Weights) -> np.ndarray:
    """x_0 of one f-gram: its token rows plus the position rows, float64 [n, d]."""
    idx = np.asarray(tokens, np.int64)
    x0 = bf16_to_f64(T_rows[idx])
    x0 = x0 + position_rows(W, idx.shape[0])
    return x0


def fgram_row(tokens, T_rows: np.ndarray, W: Weights, emulate_bf16: bool = True) -> np.ndarray:
    """F(w) for one f-gram: float64 [d] (bf16 values when emulating)."""
    x = forward_states(model_input(tokens, T_rows, W), W, emulate_bf16)
    f = layer_norm(x[-1:])[0]
    return bf16_round(f) if emulate_bf16 else f


def precompute(fgram_tok: np.ndarray, fgram_len: np.ndarray, T_rows: np.ndarray, W: Weights,
               emulate_bf16: bool = True) -> np.ndarray:
    """F rows for a list of f-grams ([N, K] padded, [N]): float64 [N, d]."""
    out = np.empty((len(fgram_len), W.m.d))
    for r, (t, n) in enumerate(zip(fgram_tok, fgram_len)):
        out[r] = fgram_row(t[:int(n)], T_rows, W, emulate_bf16)
    return out
