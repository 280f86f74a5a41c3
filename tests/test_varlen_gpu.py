"""Ragged and continued batches (scone_embed_varlen) against the oracle (GPU).

The oracle has no notion of packing or of chunks: for every sequence it
runs Algorithm 1 over the sequence's whole known prefix (history ++ chunk)
and the expected rows of the chunk are its last positions. Cases: ragged
lengths with empty and one-token sequences; equal lengths (equals
scone_embed); a long prompt fed in random chunks (chunked prefill) equals
one prefill; decode steps equal scone_decode_step; mixed prefill and
decode chunks in one launch with a slot map; error positions.
"""

import numpy as np
import pytest
import torch

import synth
import paper_2502_01637_gb300 as scone
from gpu_cases import DEV, SmallCase

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS["tiny"].scaled("varlen", B=1, L=64, d=64,
                                   quotas=((2, 4000), (3, 3000)))


@pytest.fixture(scope="module")
def case():
    c = SmallCase(W, tok=np.zeros((1, 1), np.int32))
    c.table = c.build()
    yield c
    c.table.close()


def stream_tokens(n, seed):
    return synth.zipf_tokens(W, seed, n, inject=False)


def expected_chunk(case, seq_tokens, h):
    """Oracle rows for the last len(seq_tokens) - h positions of one sequence."""
    tok = np.asarray(seq_tokens, np.int32)[None, :]
    out, row, ln, rc = case.oracle.embed(tok, case.F, case.T)
    return out[0, h:], row[0, h:], ln[0, h:], rc


def run_varlen(case, chunks, state=None, slots=None):
    lens = [len(c) for c in chunks]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    flat = np.concatenate([np.asarray(c, np.int32) for c in chunks]) if sum(lens) else \
        np.zeros(0, np.int32)
    n = flat.size
    tok = torch.from_numpy(flat).to(DEV)
    cu_d = torch.from_numpy(cu).to(DEV)
    out = torch.empty((max(n, 1), W.d), dtype=torch.int16, device=DEV)
    row = torch.empty(max(n, 1), dtype=torch.int32, device=DEV)
    ln = torch.empty(max(n, 1), dtype=torch.uint8, device=DEV)
    sl = torch.from_numpy(np.asarray(slots, np.int32)).to(DEV) if slots is not None else None
    scone.scone_embed_varlen(case.table, tok, cu_d, out[:n], state=state, seq_slot=sl,
                             row=row[:n], len=ln[:n])
    torch.cuda.synchronize()
    return (out[:n].cpu().numpy().view(np.uint16), row[:n].cpu().numpy(), ln[:n].cpu().numpy(),
            cu)


def test_ragged_fresh_sequences(case):
    lens = [0, 1, 2, 3, 37, 0, 500, 1, 64, 129, 0]
    chunks = [stream_tokens(n, 100 + k) for k, n in enumerate(lens)]
    out, row, ln, cu = run_varlen(case, chunks)
    for b, c in enumerate(chunks):
        if not len(c):
            continue
        eo, er, el, rc = expected_chunk(case, c, 0)
        sl = slice(cu[b], cu[b + 1])
        assert np.array_equal(row[sl], er.astype(np.int32)), b
        assert np.array_equal(ln[sl], el), b
        assert np.array_equal(out[sl], eo), b
    assert scone.scone_status(case.table) == 0


def test_equal_lengths_equal_dense_embed(case):
    tok = synth.query_tokens(W.scaled("varlen_dense", B=6, L=300))
    t = torch.from_numpy(tok).to(DEV)
    out_d = torch.empty((tok.size, W.d), dtype=torch.int16, device=DEV)
    row_d = torch.empty(tok.size, dtype=torch.int32, device=DEV)
    scone.scone_embed(case.table, t, out_d, row_d)
    out, row, ln, _ = run_varlen(case, list(tok))
    assert np.array_equal(row, row_d.cpu().numpy())
    assert np.array_equal(out, out_d.cpu().numpy().view(np.uint16))


def test_chunked_prefill_equals_one_prefill(case):
    """One 700-token prompt per slot, fed in random chunks (some empty);
    every chunk's rows equal the whole prompt's rows at those positions."""
    rng = np.random.default_rng(1)
    S = 5
    prompts = [stream_tokens(700, 200 + s) for s in range(S)]
    H = W.K - 1
    st = scone.scone_decode_create(case.table, np.zeros((S, H), np.int32),
                                   np.zeros(S, np.int32))
    full = [expected_chunk(case, p, 0) for p in prompts]
    pos = [0] * S
    for rnd in range(12):
        chunks = []
        for s in range(S):
            c = int(rng.integers(0, 90)) if rnd < 11 else 700 - pos[s]
            c = min(c, 700 - pos[s])
            chunks.append(prompts[s][pos[s]:pos[s] + c])
        out, row, ln, cu = run_varlen(case, chunks, state=st)
        for s in range(S):
            a, b = pos[s], pos[s] + len(chunks[s])
            sl = slice(cu[s], cu[s + 1])
            assert np.array_equal(row[sl], full[s][1][a:b].astype(np.int32)), (rnd, s)
            assert np.array_equal(ln[sl], full[s][2][a:b]), (rnd, s)
            assert np.array_equal(out[sl], full[s][0][a:b]), (rnd, s)
            pos[s] = b
    assert pos == [700] * S
    hist, hl = scone.scone_decode_get_history(st)
    for s in range(S):
        assert hl[s] == H and list(hist[s]) == list(prompts[s][-H:])
    st.close()


def test_decode_chunks_equal_decode_step(case):
    S, steps = 40, 6
    H = W.K - 1
    rng = np.random.default_rng(2)
    hist = rng.integers(0, W.vocab, size=(S, H)).astype(np.int32)
    hl = rng.integers(0, H + 1, size=S).astype(np.int32)
    new = np.stack([stream_tokens(S, 300 + k) for k in range(steps)])
    a = scone.scone_decode_create(case.table, hist, hl)
    b = scone.scone_decode_create(case.table, hist, hl)
    for k in range(steps):
        out_a = torch.empty((S, W.d), dtype=torch.int16, device=DEV)
        row_a = torch.empty(S, dtype=torch.int32, device=DEV)
        scone.scone_decode_step(a, torch.from_numpy(new[k]).to(DEV), out_a, row_a)
        out, row, ln, _ = run_varlen(case, [new[k][s:s + 1] for s in range(S)], state=b)
        assert np.array_equal(row, row_a.cpu().numpy()), k
        assert np.array_equal(out, out_a.cpu().numpy().view(np.uint16)), k
    ha, la = scone.scone_decode_get_history(a)
    hb, lb = scone.scone_decode_get_history(b)
    assert np.array_equal(la, lb)
    for s in range(S):
        assert list(ha[s][H - la[s]:]) == list(hb[s][H - lb[s]:])
    a.close()
    b.close()


def test_mixed_batch_with_slot_map(case):
    """Prefill chunks and one-token decode chunks in one launch; sequences map
    to slots out of order; slots not named keep their history."""
    S = 12
    H = W.K - 1
    st = scone.scone_decode_create(case.table, np.zeros((S, H), np.int32), np.zeros(S, np.int32))
    rng = np.random.default_rng(3)
    seqs = {s: list(stream_tokens(int(rng.integers(1, 40)), 400 + s)) for s in range(S)}
    # first batch: slots 0..11 prefill in a shuffled order
    order = rng.permutation(S)
    run_varlen(case, [np.array(seqs[s], np.int32) for s in order], state=st, slots=order)
    for rnd in range(4):
        chosen = rng.choice(S, 7, replace=False)
        chunks, slots = [], []
        for s in chosen:
            c = stream_tokens(1 if s % 2 else int(rng.integers(2, 30)), 500 + 10 * rnd + s)
            chunks.append(c)
            slots.append(int(s))
        out, row, ln, cu = run_varlen(case, chunks, state=st, slots=slots)
        for q, s in enumerate(slots):
            h = len(seqs[s])
            seqs[s] += list(chunks[q])
            eo, er, el, _ = expected_chunk(case, seqs[s], h)
            sl = slice(cu[q], cu[q + 1])
            assert np.array_equal(row[sl], er.astype(np.int32)), (rnd, s)
            assert np.array_equal(out[sl], eo), (rnd, s)
    hist, hl = scone.scone_decode_get_history(st)
    for s in range(S):
        k = int(hl[s])
        assert k == min(H, len(seqs[s]))
        assert list(hist[s][H - k:]) == seqs[s][len(seqs[s]) - k:]
    st.close()


def test_error_positions(case):
    S = 3
    H = W.K - 1
    st = scone.scone_decode_create(case.table, np.zeros((S, H), np.int32), np.zeros(S, np.int32))
    chunks = [stream_tokens(5, 600), stream_tokens(4, 601)]
    chunks[0][2] = W.vocab           # invalid token
    out, row, ln, cu = run_varlen(case, chunks, state=st, slots=[0, 7])   # slot 7 >= S
    assert ln[2] == 0 and row[2] == -1 and not out[2].any()
    sl = slice(cu[1], cu[2])
    assert (ln[sl] == 0).all() and (row[sl] == -1).all() and not out[sl].any()
    rc = scone.scone_status(case.table, raise_on_error=False)
    assert rc in (scone.SCONE_ERR_TOKEN_RANGE, scone.SCONE_ERR_INVALID_ARG)
    st.close()


def ragged_continued(w, seed, rounds=6, per_seq=400, mode=None, fgrams=None):
    """Six rounds of ragged chunks (some empty) that continue S slots, the
    last round flushing each sequence's rest; every chunk's rows match the
    oracle on the sequence's whole prefix."""
    c = SmallCase(w, fgrams=fgrams, tok=np.zeros((1, 1), np.int32))
    c.table = c.build()
    if mode is not None:
        scone.scone_table_set_copy_mode(c.table, mode)
    S, H = 6, w.K - 1
    st = scone.scone_decode_create(c.table, np.zeros((S, H), np.int32), np.zeros(S, np.int32))
    full = [synth.zipf_tokens(w, seed + s, per_seq) for s in range(S)]
    pos = [0] * S
    rng = np.random.default_rng(seed)
    matched = np.zeros(w.K + 1, np.int64)
    for rnd in range(rounds):
        chunks = []
        for s in range(S):
            n = min(int(rng.integers(0, 120)) if rnd < rounds - 1 else per_seq, per_seq - pos[s])
            chunks.append(full[s][pos[s]:pos[s] + n])
        lens = [len(x) for x in chunks]
        cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        flat = np.concatenate(chunks).astype(np.int32) if sum(lens) else np.zeros(0, np.int32)
        n = flat.size
        out = torch.empty((max(n, 1), w.d), dtype=torch.int16, device=DEV)
        row = torch.empty(max(n, 1), dtype=torch.int32, device=DEV)
        ln = torch.empty(max(n, 1), dtype=torch.uint8, device=DEV)
        scone.scone_embed_varlen(c.table, torch.from_numpy(flat).to(DEV),
                                 torch.from_numpy(cu).to(DEV), out[:n], state=st, row=row[:n],
                                 len=ln[:n])
        torch.cuda.synchronize()
        g_out = out[:n].cpu().numpy().view(np.uint16)
        g_row, g_len = row[:n].cpu().numpy(), ln[:n].cpu().numpy()
        for s in range(S):
            a, b = pos[s], pos[s] + lens[s]
            exp_out, exp_row, exp_len, rc = c.oracle.embed(
                np.asarray(full[s][:b], np.int32)[None, :], c.F, c.T)
            sl = slice(cu[s], cu[s + 1])
            assert np.array_equal(g_row[sl], exp_row[0, a:b].astype(np.int32)), (rnd, s)
            assert np.array_equal(g_len[sl], exp_len[0, a:b]), (rnd, s)
            assert np.array_equal(g_out[sl], exp_out[0, a:b]), (rnd, s)
            matched += np.bincount(exp_len[0, a:b], minlength=w.K + 1)
            pos[s] = b
    assert pos == [per_seq] * S
    assert scone.scone_status(c.table) == 0
    info = c.table.info()
    st.close()
    c.table.close()
    return matched, info


@pytest.mark.parametrize("mode", [scone.SCONE_COPY_AUTO, scone.SCONE_COPY_REGISTERS])
def test_k5_ragged_and_continued(mode):
    """K = 5 over the stress law, with phrases injected often enough that 4-
    and 5-gram matches occur (and cross chunk boundaries); AUTO walks the
    lengths over the table's suffix index, REGISTERS looks every length up."""
    w5 = synth.WORKLOADS["stress_k5"].scaled("varlen_k5", B=1, L=64, d=64,
                                             quotas=((2, 3000), (3, 3000), (4, 1500), (5, 1500)),
                                             inject_p=0.05, n_phrases=256, phrase_len=(5, 7))
    matched, info = ragged_continued(w5, 900, mode=mode)
    assert matched[4] and matched[5]
    assert info["suffix_index"] == 1


@pytest.mark.parametrize("mode", [scone.SCONE_COPY_AUTO, scone.SCONE_COPY_REGISTERS])
def test_unclosed_list_ragged_and_continued(mode):
    """A K = 4 list with half of its shorter f-grams left out, so that the
    table holds many marker slots: the walk and the register kernel both
    follow the oracle over ragged, continued chunks."""
    w = synth.Workload("varlen_unclosed", 71, 3000, 1.05, 1, 64,
                       ((2, 3000), (3, 3000), (4, 3000)), 4, 64, inject_p=0.05, n_phrases=256,
                       phrase_len=(4, 6))
    ft, fl, _ = synth.fgram_set(w)
    keep = ~((fl < 4) & (np.arange(fl.shape[0]) % 2 == 0))
    matched, info = ragged_continued(w, 1300, mode=mode, fgrams=(ft[keep], fl[keep]))
    assert info["n_markers"] > 100
    assert matched[2] and matched[4]


@pytest.mark.parametrize("name,K,vocab,slot_bytes", [
    ("k5_fmt32", 5, 300000, 32),
    ("k8_fmt32", 8, 1 << 20, 32),
    ("k8_fmt16", 8, 2000, 16),
    ("k2_fmt16", 2, 2000, 16),
])
def test_key_formats_ragged_and_continued(name, K, vocab, slot_bytes):
    """Every (key format, K bound) instance of the varlen kernel: 16- and
    32-byte slots with K up to 8, over phrase-injected streams so that long
    matches occur across chunk boundaries."""
    w = synth.Workload(name, 60 + K, vocab, 1.05, 1, 64, tuple((n, 1500) for n in range(2, K + 1)),
                       K, 64, inject_p=0.05, n_phrases=256, phrase_len=(K, K + 2))
    matched, info = ragged_continued(w, 1000 + K)
    assert info["slot_bytes"] == slot_bytes
    assert matched[2] and matched[K]


@pytest.mark.parametrize("K,mode", [(3, scone.SCONE_COPY_AUTO), (3, scone.SCONE_COPY_REGISTERS),
                                    (5, scone.SCONE_COPY_AUTO), (5, scone.SCONE_COPY_REGISTERS)])
def test_many_short_chunks_across_warps(K, mode):
    """Thousands of chunks of 0..5 tokens continuing as many slots, in three
    launches: the chunks' first K-1 positions (the readers of a slot's old
    history) fall across warp boundaries many times per launch, and each
    slot's history is rewritten in the launch that reads it. Every position
    equals the oracle on its sequence's whole prefix."""
    quotas = tuple((n, 2000) for n in range(2, K + 1))
    w = synth.Workload(f"short_chunks_k{K}", 90 + K, 2000, 1.05, 1, 64, quotas, K, 64,
                       inject_p=0.05, n_phrases=256, phrase_len=(K, K + 2))
    c = SmallCase(w, tok=np.zeros((1, 1), np.int32))
    c.table = c.build()
    scone.scone_table_set_copy_mode(c.table, mode)
    S, H, rounds = 6000, K - 1, 3
    st = scone.scone_decode_create(c.table, np.zeros((S, H), np.int32), np.zeros(S, np.int32))
    rng = np.random.default_rng(K)
    full = [synth.zipf_tokens(w, 5000 + s, 5 * rounds) for s in range(S)]
    pos = np.zeros(S, np.int64)
    for rnd in range(rounds):
        order = rng.permutation(S)                 # slots in a new order every launch
        lens = rng.integers(0, 6, S)
        chunks = [full[s][pos[s]:pos[s] + lens[k]] for k, s in enumerate(order)]
        cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        flat = np.concatenate(chunks).astype(np.int32)
        n = flat.size
        out = torch.empty((n, w.d), dtype=torch.int16, device=DEV)
        row = torch.empty(n, dtype=torch.int32, device=DEV)
        ln = torch.empty(n, dtype=torch.uint8, device=DEV)
        scone.scone_embed_varlen(c.table, torch.from_numpy(flat).to(DEV),
                                 torch.from_numpy(cu).to(DEV), out, state=st,
                                 seq_slot=torch.from_numpy(order.astype(np.int32)).to(DEV),
                                 row=row, len=ln)
        torch.cuda.synchronize()
        g_out = out.cpu().numpy().view(np.uint16)
        g_row, g_len = row.cpu().numpy(), ln.cpu().numpy()
        for k, s in enumerate(order):
            if lens[k] == 0:
                continue
            a, b = int(pos[s]), int(pos[s] + lens[k])
            e_out, e_row, e_len, _ = c.oracle.embed(np.asarray(full[s][:b], np.int32)[None, :],
                                                    c.F, c.T)
            sl = slice(cu[k], cu[k + 1])
            assert np.array_equal(g_len[sl], e_len[0, a:b]), (rnd, s)
            assert np.array_equal(g_row[sl], e_row[0, a:b].astype(np.int32)), (rnd, s)
            assert np.array_equal(g_out[sl], e_out[0, a:b]), (rnd, s)
            pos[s] = b
    hist, hlen = scone.scone_decode_get_history(st)
    for s in range(S):                         # the histories the launches left behind
        m = int(min(H, pos[s]))
        assert hlen[s] == m
        assert np.array_equal(hist[s, H - m:], np.asarray(full[s][pos[s] - m:pos[s]]))
    assert scone.scone_status(c.table) == 0
    st.close()
    c.table.close()
