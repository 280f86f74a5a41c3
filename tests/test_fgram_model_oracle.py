"""The f-gram model oracle (oracle/fgram_model.py) pinned to things other
than itself (CPU only).

Pins: bf16 rounding against torch's float32 -> bfloat16 conversion; the
rotary embedding (the non-default position option) against hand-derived
values and the relative-position property; attention against torch's
scaled_dot_product_attention and a pure-Python loop; layer norm and SiLU
against torch; the whole forward, in float64, against a second forward
assembled from torch library calls with its own unpacking of the weight
buffer, for both position schemes; the paper's padded batches (Appendix F:
f-grams padded to the longest in the batch, absolute positions) through that
library forward against the oracle's unpadded rows; special cases (no layers:
F is the layer norm of the last token's row plus the position row of the last
position), causality and head-permutation invariance.
"""

import dataclasses
import importlib
import importlib.util
import math
import os

import numpy as np
import pytest
import torch

import synth


def _load_oracle():
    path = os.environ.get("SCONE_FGRAM_ORACLE_FILE")
    if not path:
        return importlib.import_module("oracle.fgram_model")
    spec = importlib.util.spec_from_file_location("fgram_model_under_test", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


fm = _load_oracle()
TINY = synth.MODELS["tiny"]


@pytest.fixture(scope="module")
def tiny():
    packed = synth.model_weights_cpu(TINY)
    T = synth.rows_range_cpu(12345, TINY.d, 0, 300)
    return packed, fm.Weights(packed, TINY), T


def test_bf16_round_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 6, 20000),
                        [1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 0.0, 256.5]])
    x32 = x.astype(np.float32)
    want = torch.from_numpy(x32).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(fm.bf16_round(x32.astype(np.float64)), want)
    assert np.array_equal(fm.bf16_bits(want),
                          torch.from_numpy(x32).to(torch.bfloat16).view(torch.int16).numpy()
                          .view(np.uint16))


def test_rope_hand_values():
    # hd = 4: pairs (0, 2) with angle pos * 1, (1, 3) with angle pos * 10000^(-1/2) = pos / 100
    x = np.eye(4)
    r1 = fm.rope(x, np.ones(4, np.int64))
    assert np.allclose(r1[0], [math.cos(1), 0, math.sin(1), 0])
    assert np.allclose(r1[1], [0, math.cos(0.01), 0, math.sin(0.01)])
    assert np.allclose(r1[2], [-math.sin(1), 0, math.cos(1), 0])
    assert np.allclose(fm.rope(x, np.zeros(4, np.int64)), x)


def test_rope_relative_positions():
    rng = np.random.default_rng(1)
    q, k = rng.standard_normal((1, 64)), rng.standard_normal((1, 64))
    for m, n in [(0, 3), (2, 5), (7, 1)]:
        a = fm.rope(q, np.array([m])) @ fm.rope(k, np.array([n])).T
        b = fm.rope(q, np.array([m + 11])) @ fm.rope(k, np.array([n + 11])).T
        assert np.allclose(a, b)
    assert np.allclose(np.linalg.norm(fm.rope(q, np.array([9]))), np.linalg.norm(q))


@pytest.mark.parametrize("rotary", [False, True])
def test_attention_matches_torch_sdpa(rotary):
    rng = np.random.default_rng(2)
    n, H, hd = 5, 3, 8
    q, k, v = (rng.standard_normal((n, H * hd)) for _ in range(3))
    got = fm.attention(q, k, v, H, rotary)
    pos = np.arange(n)
    for h in range(H):
        sl = slice(h * hd, (h + 1) * hd)
        qh, kh = q[:, sl], k[:, sl]
        if rotary:
            qh, kh = fm.rope(qh, pos), fm.rope(kh, pos)
        vh = torch.from_numpy(v[:, sl])[None, None]
        want = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(qh)[None, None], torch.from_numpy(kh)[None, None], vh,
            is_causal=True)
        assert np.allclose(got[:, sl], want[0, 0].numpy(), atol=1e-12)


@pytest.mark.parametrize("rotary", [False, True])
def test_attention_brute_force_loops(rotary):
    rng = np.random.default_rng(3)
    n, hd = 3, 2
    q, k, v = (rng.standard_normal((n, hd)) for _ in range(3))
    got = fm.attention(q, k, v, 1, rotary)
    qr, kr = (fm.rope(q, np.arange(n)), fm.rope(k, np.arange(n))) if rotary else (q, k)
    for i in range(n):
        w = [math.exp(sum(qr[i, c] * kr[j, c] for c in range(hd)) / math.sqrt(hd))
             for j in range(i + 1)]
        for c in range(hd):
            assert abs(got[i, c] - sum(w[j] * v[j, c] for j in range(i + 1)) / sum(w)) < 1e-12


def test_layer_norm_and_silu_match_torch():
    rng = np.random.default_rng(4)
    x = rng.standard_normal((7, 96)) * 3 + 1
    want = torch.nn.functional.layer_norm(torch.from_numpy(x), (96,), eps=1e-5).numpy()
    assert np.allclose(fm.layer_norm(x), want, atol=1e-12)
    assert np.allclose(fm.silu(x), torch.nn.functional.silu(torch.from_numpy(x)).numpy())


def torch_forward_batch(fgrams, packed, T, model):
    """A second float64 forward from torch library calls, over a batch padded
    the paper's way (Appendix F): every f-gram padded after its last token to
    the batch's longest, absolute position j added to the j-th input row (or
    rotary embeddings on q and k for a rotary model), causal attention; F is
    read at each f-gram's last token. The weight buffer is unpacked here by
    index arithmetic on the documented layout."""
    d, f, H = model.d, model.ffw, model.n_heads
    hd = d // H
    w = torch.from_numpy(fm.bf16_to_f64(packed))
    B = len(fgrams)
    n_max = max(len(g) for g in fgrams)
    pad = np.zeros((B, n_max), np.int64)                    # padding token: row 0 of T
    for b, g in enumerate(fgrams):
        pad[b, :len(g)] = g
    x = torch.from_numpy(fm.bf16_to_f64(T[pad]))            # [B, n_max, d]
    layer_elems = 3 * d * d + d * d + 2 * f * d + d * f
    if model.position == "absolute":
        off = model.n_layers * layer_elems
        P = w[off:off + model.max_pos * d].reshape(model.max_pos, d)
        x = x + P[:n_max][None]
    gate_rows = torch.tensor([32 * (j // 16) + j % 16 for j in range(f)])
    up_rows = gate_rows + 16
    for layer in range(model.n_layers):
        base = layer * layer_elems
        qkv = w[base:base + 3 * d * d].reshape(3 * d, d)
        wo = w[base + 3 * d * d:base + 4 * d * d].reshape(d, d)
        gu = w[base + 4 * d * d:base + 4 * d * d + 2 * f * d].reshape(2 * f, d)
        wd = w[base + 4 * d * d + 2 * f * d:base + layer_elems].reshape(d, f)
        xn = torch.nn.functional.layer_norm(x, (d,), eps=1e-5)
        q, k, v = ((xn @ qkv[i * d:(i + 1) * d].T).reshape(B, n_max, H, hd).transpose(1, 2)
                   for i in range(3))
        if model.position == "rotary":
            pos = np.arange(n_max)
            q = torch.from_numpy(np.stack([[fm.rope(q[b, h].numpy(), pos) for h in range(H)]
                                           for b in range(B)]))
            k = torch.from_numpy(np.stack([[fm.rope(k[b, h].numpy(), pos) for h in range(H)]
                                           for b in range(B)]))
        a = torch.nn.functional.scaled_dot_product_attention(q, k, v, is_causal=True)
        x = x + a.transpose(1, 2).reshape(B, n_max, d) @ wo.T
        xn = torch.nn.functional.layer_norm(x, (d,), eps=1e-5)
        a = torch.nn.functional.silu(xn @ gu[gate_rows].T) * (xn @ gu[up_rows].T)
        x = x + a @ wd.T
    last = torch.stack([x[b, len(g) - 1] for b, g in enumerate(fgrams)])
    return torch.nn.functional.layer_norm(last, (d,), eps=1e-5).numpy()


def torch_forward(tokens, packed, T, model):
    return torch_forward_batch([list(tokens)], packed, T, model)[0]


def test_forward_matches_library_forward(tiny):
    packed, W, T = tiny
    for toks in ([5, 17], [3, 3, 9], [250, 1, 77, 8, 120]):
        got = fm.fgram_row(toks, T, W, emulate_bf16=False)
        assert np.allclose(got, torch_forward(toks, packed, T, TINY), atol=1e-9)


def test_rotary_option_matches_library_forward():
    m = dataclasses.replace(TINY, name="tiny_rotary", position="rotary")
    packed = synth.model_weights_cpu(m)
    assert packed.size == m.n_layers * m.layer_elems           # no position table
    W = fm.Weights(packed, m)
    T = synth.rows_range_cpu(12345, m.d, 0, 300)
    for toks in ([5, 17], [250, 1, 77, 8, 120]):
        got = fm.fgram_row(toks, T, W, emulate_bf16=False)
        assert np.allclose(got, torch_forward(toks, packed, T, m), atol=1e-9)


def test_padded_batches_equal_unpadded_rows(tiny):
    """Appendix F pads the f-grams of a batch to the longest one; with the
    padding after the last token and causal attention, each f-gram's row
    equals the oracle's row computed on the f-gram alone."""
    packed, W, T = tiny
    rng = np.random.default_rng(8)
    fgrams = [list(rng.integers(0, 300, n)) for n in (2, 5, 3, 8, 2, 4)]
    got = torch_forward_batch(fgrams, packed, T, TINY)
    for b, g in enumerate(fgrams):
        assert np.allclose(fm.fgram_row(g, T, W, emulate_bf16=False), got[b], atol=1e-9)


def test_positions_matter_and_come_from_P(tiny):
    """The same tokens at other positions give another row, and a model whose
    P is zero gives the rows of the model without positions."""
    packed, W, T = tiny
    a = fm.fgram_row([7, 7, 7], T, W, emulate_bf16=False)
    b = fm.fgram_row([7, 7], T, W, emulate_bf16=False)
    assert not np.allclose(a, b)
    z = packed.copy()
    z[TINY.pos_offset:] = 0
    Wz = fm.Weights(z, TINY)
    x0 = fm.model_input([3, 9, 4], T, Wz)
    assert np.array_equal(x0, fm.bf16_to_f64(T[[3, 9, 4]]))


def test_emulated_bf16_is_close_and_representable(tiny):
    _, W, T = tiny
    exact = fm.fgram_row([5, 17, 30], T, W, emulate_bf16=False)
    emu = fm.fgram_row([5, 17, 30], T, W, emulate_bf16=True)
    assert np.array_equal(fm.bf16_round(emu), emu)
    assert np.abs(emu - exact).max() < 0.1 and np.abs(emu - exact).mean() < 0.02


def test_no_layers_is_layer_norm_of_last_row_plus_its_position():
    """With no layers F = LN(T[last] + P[n-1]); with bf16 storage, byte for
    byte bf16(LN(bf16(T[last] + P[n-1])))."""
    m0 = synth.FgramModel("none", 99, 256, 4, 512, 0, max_pos=5)
    packed = synth.model_weights_cpu(m0)
    assert packed.size == 5 * 256
    P = fm.bf16_to_f64(packed).reshape(5, 256)
    W = fm.Weights(packed, m0)
    T = synth.rows_range_cpu(7, 256, 0, 10)
    for toks in ([2, 4], [1, 8, 3], [0, 0, 9, 9, 6]):
        n = len(toks)
        x = fm.bf16_to_f64(T[toks[-1]]) + P[n - 1]
        want = (x - x.mean()) / np.sqrt(x.var() + 1e-5)
        assert np.allclose(fm.fgram_row(toks, T, W, emulate_bf16=False), want, atol=1e-12)
        xb = fm.bf16_round(x)
        want_b = fm.bf16_round((xb - xb.mean()) / np.sqrt(xb.var() + 1e-5))
        assert np.array_equal(fm.bf16_bits(fm.fgram_row(toks, T, W, emulate_bf16=True)),
                              fm.bf16_bits(want_b))
    with pytest.raises(ValueError):
        fm.fgram_row([1, 2, 3, 4, 5, 6], T, W)                 # more tokens than positions


def test_causal(tiny):
    _, W, T = tiny
    x3 = fm.bf16_to_f64(T[[4, 9, 13]])
    s3 = fm.forward_states(x3, W, emulate_bf16=False)
    s2 = fm.forward_states(x3[:2], W, emulate_bf16=False)
    assert np.allclose(s3[:2], s2, atol=1e-12)
    assert not np.allclose(s3[2], fm.forward_states(x3[2:], W, emulate_bf16=False)[0])


def test_head_permutation_invariance(tiny):
    packed, W, T = tiny
    d, H = TINY.d, TINY.n_heads
    hd = d // H
    perm = np.array([2, 0, 3, 1])
    rows = np.concatenate([np.arange(p * hd, (p + 1) * hd) for p in perm])
    W2 = fm.Weights(packed, TINY)
    for L in W2.layers:
        L["q"], L["k"], L["v"] = L["q"][rows], L["k"][rows], L["v"][rows]
        L["o"] = L["o"][:, rows]
    a = fm.fgram_row([8, 2, 6], T, W, emulate_bf16=False)
    b = fm.fgram_row([8, 2, 6], T, W2, emulate_bf16=False)
    assert np.allclose(a, b, atol=1e-10)
