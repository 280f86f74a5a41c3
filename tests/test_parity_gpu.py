"""CUDA path vs the oracle, element by element, on seeded inputs (GPU).

Bit-exact throughout: row ids and lengths are integers and the outputs are
copies of stored bf16 rows, so the tolerance is zero.
"""

import itertools

import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2502_01637_gb300 as scone
from gpu_cases import DEV, SmallCase, dev_rows, run_embed

pytestmark = pytest.mark.gpu

TINY = synth.WORKLOADS["tiny"]


def assert_parity(case: SmallCase, out, row, ln):
    o_out, o_row, o_len, _ = case.expected()
    n = case.tok.size
    assert np.array_equal(ln, o_len.reshape(n)), "match lengths differ"
    assert np.array_equal(row, o_row.reshape(n).astype(np.int32)), "row ids differ"
    assert np.array_equal(out, o_out.reshape(n, -1)), "output bytes differ"


@pytest.mark.parametrize("mode", ["fused", "match+gather", "fused_noaux"])
def test_tiny_full(mode):
    case = SmallCase(TINY)
    table = case.build()
    out, row, ln = run_embed(table, case.tok, TINY.d, mode)
    assert_parity(case, out, row, ln)
    assert scone.scone_status(table) == 0
    info = table.info()
    assert info["n_fgrams"] == TINY.n_fgrams and info["slot_bytes"] == 16
    assert info["n_slots"] >= 2 * TINY.n_fgrams
    # every length occurs, so every branch of the selection ran
    assert set(np.unique(ln)) == {1, 2, 3}


@pytest.mark.parametrize("B,L", [(3, 77), (1, 1), (1, 31), (2, 33), (5, 2), (7, 129)])
def test_ragged_shapes(B, L):
    w = TINY.scaled("tiny_ragged", B=B, L=L, quotas=((2, 20000), (3, 15000)))
    case = SmallCase(w)
    table = case.build()
    for mode in ("fused", "match+gather"):
        out, row, ln = run_embed(table, case.tok, w.d, mode)
        assert_parity(case, out, row, ln)


def test_empty_batches():
    case = SmallCase(TINY.scaled("tiny_empty", B=1, L=8, quotas=((2, 100), (3, 50))))
    table = case.build()
    for B, L in ((0, 5), (3, 0), (0, 0)):
        t = torch.empty((B, L), dtype=torch.int32, device=DEV)
        out = torch.empty((0, TINY.d), dtype=torch.int16, device=DEV)
        scone.scone_embed(table, t, out)
        scone.scone_match(table, t, torch.empty(0, dtype=torch.int32, device=DEV))
    assert scone.scone_status(table) == 0


@pytest.mark.parametrize("name,K,vocab,d,quotas,inject", [
    ("k2", 2, 32000, 256, ((2, 8000),), 0.0),
    ("k4_d512", 4, 50000, 512, ((2, 6000), (3, 6000), (4, 6000)), 0.02),
    ("k5_stress", 5, 100000, 1536, ((2, 20000), (3, 20000), (4, 10000), (5, 10000)), 0.05 / 6),
    ("k5_fmt32", 5, 300000, 128, ((2, 5000), (3, 5000), (4, 5000), (5, 5000)), 0.05),
    ("k8_fmt32", 8, 1 << 20, 64, tuple((n, 2000) for n in range(2, 9)), 0.05),
    ("k7_fmt16", 7, 8192, 64, tuple((n, 2000) for n in range(2, 8)), 0.05),
    ("k3_d1024", 3, 100000, 1024, ((2, 6000), (3, 4000)), 0.0),
    ("k3_d4096", 3, 100000, 4096, ((2, 600), (3, 400)), 0.0),
])
def test_key_formats_and_widths(name, K, vocab, d, quotas, inject):
    w = synth.Workload(name, 40 + K, vocab, 1.05, 3, 700, quotas, K, d, inject_p=inject,
                       n_phrases=512 if inject else 0, phrase_len=(K, K + 2))
    case = SmallCase(w)
    table = case.build()
    info = table.info()
    bits = int(np.ceil(np.log2(vocab)))
    assert info["bits_per_token"] == bits
    assert info["slot_bytes"] == (16 if K * bits <= 92 else 32)
    out, row, ln = run_embed(table, case.tok, d)
    assert_parity(case, out, row, ln)
    assert (ln >= 2).any()
    if K in (2, 4, 5):
        assert (ln == K).any(), "longest length never matched"


@pytest.mark.parametrize("d,offset", [(100, 0), (6, 0), (3, 0), (256, 1), (8, 2)])
def test_generic_copy_widths(d, offset):
    """Rows or outputs not 16-byte aligned take the 8, 4 or 2 byte copy."""
    w = TINY.scaled(f"tiny_d{d}", B=2, L=150, d=d, quotas=((2, 4000), (3, 3000)))
    case = SmallCase(w)
    table = case.build()
    for mode in ("fused", "match+gather"):
        out, row, ln = run_embed(table, case.tok, d, mode, out_offset=offset)
        assert_parity(case, out, row, ln)


@pytest.mark.parametrize("lf", [0.1, 0.25, 0.5, 0.7, 0.85])
def test_load_factors(lf):
    w = TINY.scaled("tiny_lf", B=2, L=512)
    case = SmallCase(w)
    table = case.build(load_factor=lf)
    info = table.info()
    assert info["n_slots"] >= int(np.ceil(w.n_fgrams / lf))
    out, row, ln = run_embed(table, case.tok, w.d)
    assert_parity(case, out, row, ln)


def test_permuted_list_same_output():
    w = TINY.scaled("tiny_perm", B=2, L=300, quotas=((2, 5000), (3, 5000)))
    case = SmallCase(w)
    out, row, ln = run_embed(case.build(), case.tok, w.d)
    perm = np.random.default_rng(9).permutation(w.n_fgrams)
    case2 = SmallCase(w, fgrams=(case.fg_tok[perm], case.fg_len[perm]), tok=case.tok)
    case2.F = case.F[perm]
    out2, row2, ln2 = run_embed(case2.build(), case.tok, w.d)
    assert np.array_equal(out, out2) and np.array_equal(ln, ln2)
    assert np.array_equal(np.where(row2 >= 0, perm[np.maximum(row2, 0)], -1), row)


def test_empty_fgram_set_is_token_embedding():
    rng = np.random.default_rng(2)
    V, d = 1000, 64
    tok = rng.integers(0, V, size=(4, 100)).astype(np.int32)
    T = rng.integers(0, 2**16, size=(V, d), dtype=np.uint16)
    Td = dev_rows(T)
    table = scone.scone_table_build(np.zeros((0, 3), np.int32), np.zeros(0, np.uint8), 3, V, d,
                                    None, Td)
    out, row, ln = run_embed(table, tok, d)
    ref = torch.nn.functional.embedding(torch.from_numpy(tok.astype(np.int64)).to(DEV), Td)
    assert np.array_equal(out, ref.cpu().numpy().view(np.uint16).reshape(-1, d))
    assert (row == -1).all() and (ln == 1).all()


def test_invalid_tokens_zero_rows_and_status():
    w = TINY.scaled("tiny_bad", B=2, L=64, quotas=((2, 3000), (3, 2000)))
    tok = synth.query_tokens(w)
    tok[0, 5] = -1
    tok[0, 17] = w.vocab
    tok[1, 0] = 2**31 - 1
    tok[1, 40] = -7
    case = SmallCase(w, tok=tok)
    table = case.build()
    for mode in ("fused", "match+gather"):
        out, row, ln = run_embed(table, case.tok, w.d, mode)
        o_out, o_row, o_len, rc = case.expected()
        assert rc == oracle.ERR_TOKEN_RANGE
        assert_parity(case, out, row, ln)
        assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_TOKEN_RANGE
        assert scone.scone_status(table) == 0       # read clears it


def test_duplicate_fgrams_rejected():
    ft = np.array([[1, 2, -1], [3, 4, 5], [1, 2, 9]], np.int32)
    fl = np.array([2, 3, 2], np.uint8)
    T = dev_rows(np.zeros((10, 8), np.uint16))
    F = dev_rows(np.zeros((3, 8), np.uint16))
    with pytest.raises(scone.SconeError) as e:
        scone.scone_table_build(ft, fl, 3, 10, 8, F, T)
    assert e.value.code == scone.SCONE_ERR_DUPLICATE_FGRAM
    # the padding after the length is ignored: this list has no duplicate
    fl2 = np.array([2, 3, 3], np.uint8)
    ft2 = np.array([[1, 2, 7], [3, 4, 5], [1, 2, 9]], np.int32)
    scone.scone_table_build(ft2, fl2, 3, 10, 8, F, T).close()


def test_probe_limit_reports_and_never_hangs():
    """A cap of one bucket at load 0.85: a lookup whose key is not in its
    first bucket cannot conclude and becomes an error position (zero row,
    len 0, sticky status); every other position still matches."""
    w = TINY.scaled("tiny_probe", B=4, L=512)
    case = SmallCase(w)
    table = case.build(load_factor=0.85)
    assert table.info()["max_insert_probe"] > 0       # evictions happened at this load
    scone.scone_table_set_probe_limit(table, 1)
    out, row, ln = run_embed(table, case.tok, w.d)
    o_out, o_row, o_len, _ = case.expected()
    err = ln == 0
    assert err.any() and not err.all()
    assert (row[err] == -1).all() and (out[err] == 0).all()
    ok = ~err
    assert np.array_equal(ln[ok], o_len.reshape(-1)[ok])
    assert np.array_equal(out[ok], o_out.reshape(-1, w.d)[ok])
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_PROBE_LIMIT
    scone.scone_table_set_probe_limit(table, 2)         # back to both buckets
    out, row, ln = run_embed(table, case.tok, w.d)
    assert_parity(case, out, row, ln)
    assert scone.scone_status(table) == 0


def test_host_mapped_F():
    w = TINY.scaled("tiny_host", B=3, L=400)
    case = SmallCase(w)
    buf = scone.scone_host_alloc(case.F.nbytes)
    buf.numpy()[:] = case.F.reshape(-1)
    table = case.build(F_location=scone.SCONE_ROWS_HOST_MAPPED, F=buf.ptr)
    assert table.info()["F_location"] == scone.SCONE_ROWS_HOST_MAPPED
    for mode in ("fused", "match+gather"):
        out, row, ln = run_embed(table, case.tok, w.d, mode)
        assert_parity(case, out, row, ln)
    table.close()
    buf.free()


def test_pinned_host_tokens():
    """scone_embed reading its tokens straight from pinned host memory (the
    zero-copy input of the end-to-end path) gives the device-token result,
    including an out-of-range token's zero row and status."""
    w = TINY.scaled("tiny_pinned", B=5, L=333)
    case = SmallCase(w)
    case.tok[3, 17] = w.vocab + 5
    table = case.build()
    host = torch.from_numpy(case.tok).pin_memory()
    out = torch.empty((case.tok.size, w.d), dtype=torch.int16, device=DEV)
    row = torch.empty(case.tok.size, dtype=torch.int32, device=DEV)
    ln = torch.empty(case.tok.size, dtype=torch.uint8, device=DEV)
    scone.scone_embed(table, host, out, row, ln)
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_TOKEN_RANGE
    assert_parity(case, out.cpu().numpy().view(np.uint16), row.cpu().numpy(), ln.cpu().numpy())
    with pytest.raises(ValueError):
        scone.scone_embed(table, torch.from_numpy(case.tok), out)   # pageable: refused
    table.close()


# ------------------------------------------------------------------ decode
def _decode_case(K, S, steps, vocab=2000, d=96, seed=0):
    rng = np.random.default_rng(seed)
    H = K - 1
    full = (rng.zipf(1.3, size=(S, H + steps)) % vocab).astype(np.int32)
    # f-grams: windows of the sequences themselves (so long matches occur) + random ones
    fg = set()
    for s in range(S):
        for p in range(full.shape[1]):
            n = int(rng.integers(2, K + 1))
            if p + n <= full.shape[1] and rng.random() < 0.4:
                fg.add(tuple(full[s, p:p + n].tolist()))
    for _ in range(500):
        n = int(rng.integers(2, K + 1))
        fg.add(tuple(rng.integers(0, vocab, size=n).tolist()))
    fg = sorted(fg)
    ft = np.full((len(fg), K), -1, np.int32)
    fl = np.array([len(g) for g in fg], np.uint8)
    for r, g in enumerate(fg):
        ft[r, :len(g)] = g
    hl = rng.integers(0, H + 1, size=S).astype(np.int32)
    hl[:3] = [0, H, min(1, H)]
    hist = rng.integers(0, vocab, size=(S, H)).astype(np.int32)   # ignored entries: valid ids
    for s in range(S):
        if hl[s]:
            hist[s, H - hl[s]:] = full[s, H - hl[s]:H]
    new = np.ascontiguousarray(full[:, H:].T)
    F = rng.integers(0, 2**16, size=(len(fg), d), dtype=np.uint16)
    T = rng.integers(0, 2**16, size=(vocab, d), dtype=np.uint16)
    return ft, fl, hist, hl, new, F, T


@pytest.mark.parametrize("K,S,vocab", [(3, 100, 2000), (5, 70, 2000), (2, 33, 2000),
                                       (8, 40, 2000), (6, 40, 1 << 20)])
def test_decode_steps_match_oracle(K, S, vocab):
    steps, d = 12, 96
    ft, fl, hist, hl, new, F, T = _decode_case(K, S, steps, vocab, d, seed=K)
    new[3, 5] = -4            # an invalid token mid-stream
    new[7, 0] = vocab
    o = oracle.Oracle(ft, fl, K, vocab)
    o_out, o_row, o_len, rc = o.decode(hist, hl, new, F, T)
    assert rc == oracle.ERR_TOKEN_RANGE
    table = scone.scone_table_build(ft, fl, K, vocab, d, dev_rows(F), dev_rows(T))
    st = scone.scone_decode_create(table, hist, hl)
    new_d = torch.from_numpy(new).to(DEV)
    out = torch.empty((S, d), dtype=torch.int16, device=DEV)
    row = torch.empty(S, dtype=torch.int32, device=DEV)
    ln = torch.empty(S, dtype=torch.uint8, device=DEV)
    for k in range(steps):
        scone.scone_decode_step(st, new_d[k], out, row, ln)
        assert np.array_equal(ln.cpu().numpy(), o_len[k]), k
        assert np.array_equal(row.cpu().numpy(), o_row[k].astype(np.int32)), k
        assert np.array_equal(out.cpu().numpy().view(np.uint16), o_out[k]), k
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_TOKEN_RANGE
    h2, hl2 = scone.scone_decode_get_history(st)
    H = K - 1
    assert (hl2 == np.minimum(hl + steps, H)).all()
    if H:
        assert np.array_equal(h2[:, H - min(H, steps):], new.T[:, steps - min(H, steps):])
    assert set(np.unique(o_len)) >= {0, 1, 2}


def test_decode_pinned_host_tokens():
    """Decode steps reading their new tokens from pinned host memory give the
    oracle's rows, as with device tokens (the zero-copy input of the serving
    loop)."""
    K, S, steps, d = 3, 64, 8, 96
    ft, fl, hist, hl, new, F, T = _decode_case(K, S, steps, 2000, d, seed=21)
    o = oracle.Oracle(ft, fl, K, 2000)
    o_out, o_row, o_len, _ = o.decode(hist, hl, new, F, T)
    table = scone.scone_table_build(ft, fl, K, 2000, d, dev_rows(F), dev_rows(T))
    st = scone.scone_decode_create(table, hist, hl)
    host_new = torch.from_numpy(np.ascontiguousarray(new)).pin_memory()
    out = torch.empty((S, d), dtype=torch.int16, device=DEV)
    row = torch.empty(S, dtype=torch.int32, device=DEV)
    for k in range(steps):
        scone.scone_decode_step(st, host_new[k], out, row)
        torch.cuda.synchronize()
        assert np.array_equal(row.cpu().numpy(), o_row[k].astype(np.int32)), k
        assert np.array_equal(out.cpu().numpy().view(np.uint16), o_out[k]), k
    assert scone.scone_status(table) == 0
    with pytest.raises(ValueError):
        scone.scone_decode_step(st, torch.from_numpy(np.ascontiguousarray(new[0])), out)
    st.close()
    table.close()


def test_decode_equals_prefill_on_device():
    K, S, steps, vocab, d = 3, 64, 20, 2000, 64
    ft, fl, hist, hl, new, F, T = _decode_case(K, S, steps, vocab, d, seed=11)
    hl[:] = 0
    table = scone.scone_table_build(ft, fl, K, vocab, d, dev_rows(F), dev_rows(T))
    st = scone.scone_decode_create(table, hist, hl)
    new_d = torch.from_numpy(new).to(DEV)
    outs = []
    out = torch.empty((S, d), dtype=torch.int16, device=DEV)
    for k in range(steps):
        scone.scone_decode_step(st, new_d[k], out)
        outs.append(out.clone())
    dec = torch.stack(outs, 1).cpu().numpy().view(np.uint16)     # [S, steps, d]
    pre, _, _ = run_embed(table, np.ascontiguousarray(new.T), d)
    assert np.array_equal(dec.reshape(-1, d), pre)


# ---------------------------------------------------- bulk (TMA) row copies
@pytest.mark.parametrize("name,K,vocab,d,B,L,quotas", [
    ("bulk_tiny", 3, 32000, 256, 4, 512, ((2, 60000), (3, 40000))),
    ("bulk_d2048_ragged", 3, 100000, 2048, 3, 1001, ((2, 30000), (3, 20000))),
    ("bulk_k5_d1536", 5, 100000, 1536, 2, 900, ((2, 9000), (3, 9000), (4, 4000), (5, 4000))),
    ("bulk_d4096", 3, 100000, 4096, 2, 333, ((2, 3000), (3, 2000))),
    ("bulk_one_row", 3, 1000, 2048, 1, 1, ((2, 10), (3, 10))),
])
def test_bulk_copy_parity(name, K, vocab, d, B, L, quotas):
    w = synth.Workload(name, 60 + K, vocab, 1.1, B, L, quotas, K, d)
    case = SmallCase(w)
    table = case.build()
    scone.scone_table_set_copy_mode(table, scone.SCONE_COPY_BULK)
    out, row, ln = run_embed(table, case.tok, d)
    assert_parity(case, out, row, ln)
    assert scone.scone_status(table) == 0


def test_bulk_copy_error_positions_get_zero_rows():
    w = TINY.scaled("bulk_bad", B=3, L=300, quotas=((2, 3000), (3, 2000)))
    tok = synth.query_tokens(w)
    tok[0, 3] = -1
    tok[2, 299] = w.vocab + 5
    case = SmallCase(w, tok=tok)
    table = case.build()
    scone.scone_table_set_copy_mode(table, scone.SCONE_COPY_BULK)
    out, row, ln = run_embed(table, case.tok, w.d)
    assert_parity(case, out, row, ln)
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_TOKEN_RANGE


def test_bulk_copy_refuses_ineligible_calls():
    w = TINY.scaled("bulk_inel", B=1, L=64, quotas=((2, 300), (3, 200)))
    case = SmallCase(w)
    table = case.build()
    scone.scone_table_set_copy_mode(table, scone.SCONE_COPY_BULK)
    t = torch.from_numpy(case.tok).to(DEV)
    buf = torch.empty(w.B * w.L * w.d + 1, dtype=torch.int16, device=DEV)
    with pytest.raises(scone.SconeError) as e:
        scone.scone_embed(table, t, buf[1:])          # output not 16-byte aligned
    assert e.value.code == scone.SCONE_ERR_UNSUPPORTED
    with pytest.raises(scone.SconeError):
        scone.scone_table_set_copy_mode(table, 7)
    scone.scone_table_set_copy_mode(table, scone.SCONE_COPY_REGISTERS)
    out, row, ln = run_embed(table, case.tok, w.d, out_offset=1)
    assert_parity(case, out, row, ln)


# ------------------------------------------- separate match and copy warps
SPLIT_CASES = [
    ("split_k3", 3, 32000, 256, 4, 512, ((2, 60000), (3, 40000)), 0.0),
    ("split_k5_d1536", 5, 100000, 1536, 3, 1001, ((2, 9000), (3, 9000), (4, 4000), (5, 4000)),
     0.05 / 6),
    ("split_k5_fmt32", 5, 300000, 128, 3, 700, ((2, 5000), (3, 5000), (4, 5000), (5, 5000)), 0.05),
    ("split_k8_fmt32", 8, 1 << 20, 64, 3, 700, tuple((n, 2000) for n in range(2, 9)), 0.05),
    ("split_k7_fmt16", 7, 8192, 64, 2, 333, tuple((n, 2000) for n in range(2, 8)), 0.05),
    ("split_one_row", 5, 1000, 2048, 1, 1, ((2, 10), (3, 10), (4, 10), (5, 10)), 0.0),
    ("split_ragged_tail", 5, 100000, 1536, 1, 33 * 8 * 40 + 7,
     ((2, 6000), (3, 6000), (4, 3000), (5, 3000)), 0.05 / 6),
]


@pytest.mark.parametrize("mode", ["split", "pipelined"])
@pytest.mark.parametrize("name,K,vocab,d,B,L,quotas,inject", SPLIT_CASES)
def test_split_copy_parity(name, K, vocab, d, B, L, quotas, inject, mode):
    """SCONE_COPY_SPLIT (match warps hand row addresses to copy warps through
    a shared-memory ring) and SCONE_COPY_PIPELINED (the next tile's match
    interleaved into the current tile's copy; other key formats and widths
    take the register kernel): bit-exact against the oracle, for both key
    formats, ragged tile tails and a single-row batch."""
    w = synth.Workload(name, 80 + K, vocab, 1.05, B, L, quotas, K, d, inject_p=inject,
                       n_phrases=512 if inject else 0, phrase_len=(K, K + 2))
    case = SmallCase(w)
    table = case.build()
    scone.scone_table_set_copy_mode(table, {"split": scone.SCONE_COPY_SPLIT,
                                            "pipelined": scone.SCONE_COPY_PIPELINED}[mode])
    for offset in (0, 1):                    # 16-byte and 2-byte copy widths
        out, row, ln = run_embed(table, case.tok, d, out_offset=offset)
        assert_parity(case, out, row, ln)
    out2, _, _ = run_embed(table, case.tok, d, mode="fused_noaux")
    assert np.array_equal(out, out2)
    assert scone.scone_status(table) == 0


@pytest.mark.parametrize("mode", [3, 4])          # SCONE_COPY_SPLIT, SCONE_COPY_PIPELINED
def test_split_copy_error_positions_get_zero_rows(mode):
    w = TINY.scaled("split_bad", B=3, L=300, quotas=((2, 3000), (3, 2000)))
    tok = synth.query_tokens(w)
    tok[0, 3] = -1
    tok[2, 299] = w.vocab + 5
    tok[1, 40] = w.vocab                       # also inside another position's window
    case = SmallCase(w, tok=tok)
    table = case.build()
    scone.scone_table_set_copy_mode(table, mode)
    out, row, ln = run_embed(table, case.tok, w.d)
    assert_parity(case, out, row, ln)
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_TOKEN_RANGE


def test_pipelined_probe_limit_reports_and_zero_rows():
    """With one bucket per lookup allowed, the stages report the probe-limit
    error exactly where the register kernel does."""
    w = TINY.scaled("pipe_probe", B=4, L=400, quotas=((2, 30000), (3, 20000)))
    case = SmallCase(w)
    table = case.build(load_factor=0.85)
    scone.scone_table_set_probe_limit(table, 1)
    ref = run_embed(table, case.tok, w.d)
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_PROBE_LIMIT
    scone.scone_table_set_copy_mode(table, scone.SCONE_COPY_PIPELINED)
    got = run_embed(table, case.tok, w.d)
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_PROBE_LIMIT
    for a, b in zip(ref, got):
        assert np.array_equal(a, b)
    assert (ref[2] == 0).any()


@pytest.mark.parametrize("K,host_F", [(3, False), (5, False), (3, True), (5, True)])
def test_decode_bulk_row_copies(K, host_F):
    """SCONE_COPY_BULK decode steps move each row by TMA bulk copies (global or
    host-mapped F -> shared -> output); rows, lengths and bytes equal the
    oracle's, including the zero rows of invalid tokens."""
    S, steps, vocab, d = 70, 10, 2000, 128          # 256-byte rows
    ft, fl, hist, hl, new, F, T = _decode_case(K, S, steps, vocab, d, seed=30 + K)
    new[4, 9] = -2
    o = oracle.Oracle(ft, fl, K, vocab)
    o_out, o_row, o_len, _ = o.decode(hist, hl, new, F, T)
    buf = None
    if host_F:
        buf = scone.scone_host_alloc(F.nbytes)
        buf.numpy(np.uint16)[:F.size] = F.reshape(-1)
        table = scone.scone_table_build(ft, fl, K, vocab, d, buf.ptr, dev_rows(T),
                                        F_location=scone.SCONE_ROWS_HOST_MAPPED)
    else:
        table = scone.scone_table_build(ft, fl, K, vocab, d, dev_rows(F), dev_rows(T))
    scone.scone_table_set_copy_mode(table, scone.SCONE_COPY_BULK)
    st = scone.scone_decode_create(table, hist, hl)
    new_d = torch.from_numpy(new).to(DEV)
    out = torch.empty((S, d), dtype=torch.int16, device=DEV)
    row = torch.empty(S, dtype=torch.int32, device=DEV)
    ln = torch.empty(S, dtype=torch.uint8, device=DEV)
    for k in range(steps):
        out.fill_(-1)
        scone.scone_decode_step(st, new_d[k], out, row, ln)
        assert np.array_equal(ln.cpu().numpy(), o_len[k]), k
        assert np.array_equal(row.cpu().numpy(), o_row[k].astype(np.int32)), k
        assert np.array_equal(out.cpu().numpy().view(np.uint16), o_out[k]), k
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_TOKEN_RANGE
    st.close()
    table.close()
    if buf is not None:
        buf.free()


def test_default_stream_is_the_current_stream():
    """Calls without a stream argument enqueue on torch's current stream, also
    inside a stream context."""
    assert scone._stream(None) == torch.cuda.current_stream().cuda_stream
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        assert scone._stream(None) == s.cuda_stream
    assert scone._stream(None) == torch.cuda.current_stream().cuda_stream


# ------------------------------------------------- suffix index and the walk
def _unclosed_case(K, vocab, d, B, L, drop, seed, bad=()):
    """A workload whose shorter f-grams are partly dropped from the list, so
    that many suffixes of the longer ones are not f-grams (marker slots)."""
    quotas = tuple((n, 6000) for n in range(2, K + 1))
    w = synth.Workload(f"unclosed_k{K}", 60 + K, vocab, 1.05, B, L, quotas, K, d, inject_p=0.05,
                       n_phrases=512, phrase_len=(K, K + 2))
    ft, fl, _ = synth.fgram_set(w)
    keep = ~((fl < K) & (np.random.default_rng(seed).random(fl.shape[0]) < drop))
    tok = synth.query_tokens(w)
    for (b, i, x) in bad:
        tok[b, i] = x
    return SmallCase(w, fgrams=(ft[keep], fl[keep]), tok=tok)


@pytest.mark.parametrize("K,vocab,d,B,L,drop", [
    (5, 3000, 512, 5, 20011, 0.6),      # warps hold two tiles: rounds inside the copy
    (4, 3000, 256, 3, 9001, 0.9),
    (3, 3000, 256, 10, 20011, 0.7),
])
def test_suffix_walk_on_unclosed_lists(K, vocab, d, B, L, drop):
    """The table's marker count is the host index's; the walk over the lengths
    (AUTO for K = 4, 5 and PIPELINED) and the kernels that look every length
    up (REGISTERS, SPLIT) all give the oracle's rows, lengths and bytes."""
    case = _unclosed_case(K, vocab, d, B, L, drop, seed=K)
    _, _, ml = scone.scone_fgram_suffix_index(case.fg_tok, case.fg_len, K)
    assert len(ml) > 100
    table = case.build()
    info = table.info()
    assert info["n_markers"] == len(ml)
    assert info["n_slots"] >= int(np.ceil((info["n_fgrams"] + len(ml)) / 0.5))
    o_out, o_row, o_len, _ = case.expected()
    n = case.tok.size
    for mode in (scone.SCONE_COPY_AUTO, scone.SCONE_COPY_PIPELINED, scone.SCONE_COPY_REGISTERS,
                 scone.SCONE_COPY_SPLIT):
        scone.scone_table_set_copy_mode(table, mode)
        out, row, ln = run_embed(table, case.tok, d)
        assert np.array_equal(ln, o_len.reshape(n)), mode
        assert np.array_equal(row, o_row.reshape(n).astype(np.int32)), mode
        assert np.array_equal(out, o_out.reshape(n, d)), mode
        out2, _, _ = run_embed(table, case.tok, d, mode="fused_noaux")
        assert np.array_equal(out2, out)
    assert (o_len.reshape(n) == K).any()
    assert scone.scone_status(table) == 0


def test_suffix_walk_error_positions():
    """Invalid tokens (at a position, and inside later positions' windows)
    end the walk as they end the staged match: zero rows, len 0, status."""
    bad = ((0, 3, -1), (1, 40, 3000), (2, 20010, 3005), (4, 0, -7), (3, 33, 2999))
    case = _unclosed_case(5, 3000, 512, 5, 20011, 0.6, seed=5, bad=bad)
    table = case.build()
    assert table.info()["n_markers"] > 0
    out, row, ln = run_embed(table, case.tok, 512)
    assert_parity(case, out, row, ln)
    assert (ln == 0).sum() == 4
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_TOKEN_RANGE


# ------------------------------------------------- pre-scan staged through HBM
def test_prescan_staged_equals_oracle():
    """scone_prescan on a corpus in pinned host memory, staged through HBM in
    chunks of whole sequences (default size, several chunks with a short last
    one, one sequence per chunk when a chunk is shorter than a sequence, and
    no len output): the oracle's rows and lengths, the same as scone_match on
    the host addresses."""
    w = TINY.scaled("prescan_staged", B=37, L=1000)
    case = SmallCase(w)
    table = case.build()
    n = case.tok.size
    corpus = scone.scone_host_alloc(n * 4)
    corpus.numpy(np.int32)[:n] = case.tok.reshape(-1)
    rows, lens = scone.scone_host_alloc(n * 4), scone.scone_host_alloc(n)
    _, o_row, o_len, _ = case.expected()
    for chunk in (0, 5000, 999, 1000):
        rows.numpy(np.int32)[:n] = -7
        lens.numpy(np.uint8)[:n] = 99
        scone.scone_prescan(table, corpus, w.B, w.L, rows, lens, chunk_tokens=chunk)
        assert np.array_equal(rows.numpy(np.int32)[:n], o_row.reshape(-1).astype(np.int32)), chunk
        assert np.array_equal(lens.numpy(np.uint8)[:n], o_len.reshape(-1)), chunk
    rows.numpy(np.int32)[:n] = -7
    scone.scone_prescan(table, corpus, w.B, w.L, rows, None, chunk_tokens=7000)
    assert np.array_equal(rows.numpy(np.int32)[:n], o_row.reshape(-1).astype(np.int32))
    zc_rows, zc_lens = scone.scone_host_alloc(n * 4), scone.scone_host_alloc(n)
    lib = scone.load_library()
    assert lib.scone_match(table.handle, corpus.ptr, w.B, w.L, zc_rows.ptr, zc_lens.ptr,
                           torch.cuda.current_stream().cuda_stream) == 0
    torch.cuda.synchronize()
    assert np.array_equal(zc_rows.numpy(np.int32)[:n], rows.numpy(np.int32)[:n])
    assert scone.scone_status(table) == 0
    lib_inv = scone.SCONE_ERR_INVALID_ARG
    assert lib.scone_prescan(table.handle, corpus.ptr, w.B, 0, rows.ptr, None, 0, None) == lib_inv
    assert lib.scone_prescan(table.handle, None, w.B, w.L, rows.ptr, None, 0, None) == lib_inv
    for b in (corpus, rows, lens, zc_rows, zc_lens):
        b.free()
    table.close()


def test_status_reports_the_first_error_once():
    """scone_status returns the first device-detected error since the last
    call and clears it; with no error it returns 0 without launching anything
    (the kernels that record an error also write it to the table's host-mapped
    mirror, which scone_status reads after the sync)."""
    w = TINY.scaled("status_once", B=2, L=300, quotas=((2, 3000), (3, 2000)))
    tok = synth.query_tokens(w)
    bad = tok.copy()
    bad[1, 7] = w.vocab + 3
    case = SmallCase(w, tok=tok)
    table = case.build()
    for _ in range(2):
        out, row, ln = run_embed(table, tok, w.d)
        assert scone.scone_status(table) == 0
        assert_parity(case, out, row, ln)
        run_embed(table, bad, w.d)
        assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_TOKEN_RANGE
        assert scone.scone_status(table) == 0            # cleared by the call before
        assert scone.scone_status(table) == 0
    # an error in a decode step reaches the same word
    st = scone.scone_decode_create(table, np.zeros((4, 2), np.int32), np.zeros(4, np.int32))
    new = torch.tensor([1, 2, -5, 3], dtype=torch.int32, device=DEV)
    out = torch.empty((4, w.d), dtype=torch.int16, device=DEV)
    scone.scone_decode_step(st, new, out)
    assert scone.scone_status(table, raise_on_error=False) == scone.SCONE_ERR_TOKEN_RANGE
    assert scone.scone_status(table) == 0
    st.close()
    table.close()
