"""Parity at the workloads' full sizes, in the launch configuration the
benchmark times (GPU).

Every position of the full batch runs through the CUDA path, and the oracle
of Algorithm 1 answers every position too: row ids and lengths are compared
element by element, and every output row is compared with F[row] or
T[token] gathered (by torch, on the device) at the ORACLE's row ids. A sample
of positions is also compared with rows made by the host-side generator,
which ties the device copies of F and T to their seeded definition.
"""

import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2502_01637_gb300 as scone
from gpu_cases import DEV, gpu_rows

pytestmark = pytest.mark.gpu


def sample_positions(B, L, K, n_random, seed):
    rng = np.random.default_rng(seed)
    starts = np.arange(B, dtype=np.int64) * L
    pos = [rng.choice(B * L, size=min(n_random, B * L), replace=False),
           starts, starts + 1, starts + K - 1, starts + L - 1,    # sequence edges
           np.arange(min(B * L, 300)),                            # the first tiles
           np.arange(max(0, B * L - 300), B * L)]                 # the ragged end
    return np.unique(np.concatenate(pos))


def check_sampled(w, tok, row, ln, out, pos):
    o = oracle.Oracle(*synth.fgram_set(w)[:2], w.K, w.vocab)
    o_row, o_len, rc = o.select_at(tok, pos)
    assert rc == 0
    assert np.array_equal(ln[pos], o_len), "lengths differ from the oracle"
    assert np.array_equal(row[pos], o_row.astype(np.int32)), "rows differ from the oracle"
    flat_tok = tok.reshape(-1)[pos]
    exp = np.empty((pos.shape[0], w.d), np.uint16)
    hit = o_row >= 0
    exp[hit] = synth.rows_cpu(synth.F_seed(w), w.d, o_row[hit])
    exp[~hit] = synth.rows_cpu(synth.T_seed(w), w.d, flat_tok[~hit])
    got = out[torch.from_numpy(pos).to(DEV)].cpu().numpy().view(np.uint16)
    assert np.array_equal(got, exp), "output bytes differ from the oracle's rows"


def check_all_positions(w, tok, tok_d, row_d, ln_d, out, F, T, fgrams=None):
    """Every position against the oracle: rows and lengths element by
    element, output rows against the rows at the oracle's ids."""
    o = oracle.Oracle(*(fgrams if fgrams is not None else synth.fgram_set(w)[:2]), w.K, w.vocab)
    o_row, o_len, _, rc = o.select(tok)
    assert rc == 0
    o_row, o_len = o_row.reshape(-1), o_len.reshape(-1)
    row, ln = row_d.cpu().numpy(), ln_d.cpu().numpy()
    bad = np.flatnonzero((row != o_row) | (ln != o_len))
    assert bad.size == 0, (f"{bad.size} positions differ from the oracle, first at {bad[0]}: "
                           f"row {row[bad[0]]} len {ln[bad[0]]} vs oracle {o_row[bad[0]]} "
                           f"{o_len[bad[0]]}")
    r64 = torch.from_numpy(o_row).to(DEV)
    hit = r64 >= 0
    exp = T.index_select(0, tok_d.reshape(-1).to(torch.int64))
    idx = torch.nonzero(hit).reshape(-1)
    exp[idx] = F.index_select(0, r64[idx])
    eq = (out == exp).all(dim=1)
    n_bad = int((~eq).sum())
    assert n_bad == 0, f"{n_bad} output rows differ from the rows at the oracle's ids"
    return np.bincount(o_len, minlength=w.K + 1)


@pytest.mark.parametrize("name", ["prefill_1b", "large_hbm", "stress_k5"])
def test_fullsize_prefill(name):
    w = synth.WORKLOADS[name]
    fg_tok, fg_len, _ = synth.fgram_set(w)
    tok = synth.query_tokens(w)
    F = gpu_rows(synth.F_seed(w), w.n_fgrams, w.d)
    T = gpu_rows(synth.T_seed(w), w.vocab, w.d)
    table = scone.scone_table_build(fg_tok, fg_len, w.K, w.vocab, w.d, F, T,
                                    load_factor=w.load_factor)
    tok_d = torch.from_numpy(tok).to(DEV)
    n = tok.size
    out = torch.empty((n, w.d), dtype=torch.int16, device=DEV)
    row_d = torch.empty(n, dtype=torch.int32, device=DEV)
    ln_d = torch.empty(n, dtype=torch.uint8, device=DEV)
    scone.scone_embed(table, tok_d, out, row_d, ln_d)          # AUTO, as the benchmark runs
    assert scone.scone_status(table) == 0
    hist = check_all_positions(w, tok, tok_d, row_d, ln_d, out, F, T)
    assert (hist[1:] > 0).all(), f"some length never occurs: {hist}"
    # the same launch without the optional outputs writes the same rows
    out2 = torch.empty_like(out)
    scone.scone_embed(table, tok_d, out2)
    assert torch.equal(out, out2)
    pos = sample_positions(w.B, w.L, w.K, 6000, seed=len(name))
    check_sampled(w, tok, row_d.cpu().numpy(), ln_d.cpu().numpy(), out, pos)
    table.close()


def test_fullsize_stress_k5_with_markers():
    """stress_k5 with every third f-gram shorter than K left out of the list,
    so that the table's suffix index holds hundreds of thousands of marker
    slots (suffixes of listed f-grams that are not listed): every position of
    the full batch, through the walk the benchmark's kernel takes, against the
    oracle of the shortened list."""
    w = synth.WORKLOADS["stress_k5"]
    fg_tok, fg_len, _ = synth.fgram_set(w)
    keep = ~((fg_len < w.K) & (np.arange(fg_len.shape[0]) % 3 == 0))
    ft, fl = fg_tok[keep], fg_len[keep]
    F_all = gpu_rows(synth.F_seed(w), w.n_fgrams, w.d)
    F = F_all.index_select(0, torch.from_numpy(np.flatnonzero(keep)).to(DEV))
    del F_all
    T = gpu_rows(synth.T_seed(w), w.vocab, w.d)
    table = scone.scone_table_build(ft, fl, w.K, w.vocab, w.d, F, T, load_factor=w.load_factor)
    info = table.info()
    assert info["suffix_index"] == 1 and info["n_markers"] > 100_000
    tok = synth.query_tokens(w)
    tok_d = torch.from_numpy(tok).to(DEV)
    n = tok.size
    out = torch.empty((n, w.d), dtype=torch.int16, device=DEV)
    row_d = torch.empty(n, dtype=torch.int32, device=DEV)
    ln_d = torch.empty(n, dtype=torch.uint8, device=DEV)
    scone.scone_embed(table, tok_d, out, row_d, ln_d)          # AUTO: the walk
    assert scone.scone_status(table) == 0
    hist = check_all_positions(w, tok, tok_d, row_d, ln_d, out, F, T, fgrams=(ft, fl))
    assert (hist[1:] > 0).all(), f"some length never occurs: {hist}"
    table.close()


def test_fullsize_mixed_serving():
    """The serving batch the benchmark's mixed_serving times (65,536 tokens:
    48 ragged prompt chunks and 512 one-token decode chunks, each continuing
    one of 2,048 decode-state slots, prefill_1b's table), two batches in a row
    so the second continues the histories the first left. Every position
    against the oracle run over each sequence's whole known prefix (its slot's
    history ++ its chunk): rows, lengths, and output rows at the oracle's ids."""
    import bench

    w = synth.WORKLOADS["prefill_1b"]
    fg_tok, fg_len, _ = synth.fgram_set(w)
    F = gpu_rows(synth.F_seed(w), w.n_fgrams, w.d)
    T = gpu_rows(synth.T_seed(w), w.vocab, w.d)
    table = scone.scone_table_build(fg_tok, fg_len, w.K, w.vocab, w.d, F, T)
    S, H = 2048, w.K - 1
    hist = synth.query_tokens(w.scaled("mixed_hist", B=S, L=H))
    state = scone.scone_decode_create(table, hist, np.full(S, H, np.int32))
    o = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab)
    known = {s: list(hist[s]) for s in range(S)}          # each slot's tokens so far
    for k in range(2):
        tok, cu, slots = bench.mixed_batch(w, k)
        n = tok.size
        out = torch.empty((n, w.d), dtype=torch.int16, device=DEV)
        row_d = torch.empty(n, dtype=torch.int32, device=DEV)
        ln_d = torch.empty(n, dtype=torch.uint8, device=DEV)
        scone.scone_embed_varlen(table, torch.from_numpy(tok).to(DEV),
                                 torch.from_numpy(cu).to(DEV), out, state=state,
                                 seq_slot=torch.from_numpy(slots).to(DEV), row=row_d, len=ln_d)
        assert scone.scone_status(table) == 0
        o_row = np.empty(n, np.int64)
        o_len = np.empty(n, np.uint8)
        for b in range(cu.size - 1):
            chunk = tok[cu[b]:cu[b + 1]]
            if chunk.size == 0:
                continue
            seq = np.asarray(known[int(slots[b])] + chunk.tolist(), np.int32)[None, :]
            r, l_, _, rc = o.select(seq)
            assert rc == 0
            h = seq.shape[1] - chunk.size
            o_row[cu[b]:cu[b + 1]] = r[0, h:]
            o_len[cu[b]:cu[b + 1]] = l_[0, h:]
            known[int(slots[b])] = seq[0].tolist()[-H:]
        row, ln = row_d.cpu().numpy(), ln_d.cpu().numpy()
        bad = np.flatnonzero((row != o_row) | (ln != o_len))
        assert bad.size == 0, f"batch {k}: {bad.size} positions differ, first at {bad[0]}"
        r64 = torch.from_numpy(o_row).to(DEV)
        exp = T.index_select(0, torch.from_numpy(tok).to(DEV).to(torch.int64))
        idx = torch.nonzero(r64 >= 0).reshape(-1)
        exp[idx] = F.index_select(0, r64[idx])
        assert bool((out == exp).all()), f"batch {k}: output rows differ"
        assert (o_len == 3).any() and (o_len == 1).any()
    state.close()
    table.close()


def test_fullsize_offload_decode():
    """2e7 f-grams, F (82 GB) in host-pinned mapped memory; 512 sequences x 256
    steps. Rows and lengths of every step are checked against the oracle (decode
    is Algorithm 1 on prefix + new tokens), and the output bytes of all 512
    sequences on 16 steps spread over the run against the rows at the
    oracle's ids, made by the host-side generator."""
    w = synth.WORKLOADS["offload_decode"]
    fg_tok, fg_len, _ = synth.fgram_set(w)
    nbytes = w.n_fgrams * w.d * 2
    try:
        buf = scone.scone_host_alloc(nbytes)
    except scone.SconeError as e:
        pytest.fail(f"host-pinned allocation of {nbytes / 1e9:.1f} GB failed: {e}")
    stream = torch.cuda.current_stream().cuda_stream
    synth.rows_gpu(synth.F_seed(w), w.d, 0, w.n_fgrams, buf.ptr, stream)
    T = gpu_rows(synth.T_seed(w), w.vocab, w.d)
    table = scone.scone_table_build(fg_tok, fg_len, w.K, w.vocab, w.d, buf.ptr, T,
                                    F_location=scone.SCONE_ROWS_HOST_MAPPED)
    hist, hl, new = synth.decode_inputs(w)
    st = scone.scone_decode_create(table, hist, hl)
    S, steps = w.dec_S, w.dec_steps
    new_d = torch.from_numpy(new).to(DEV)
    rows = torch.empty((steps, S), dtype=torch.int32, device=DEV)
    lens = torch.empty((steps, S), dtype=torch.uint8, device=DEV)
    checked = np.unique(np.concatenate([np.arange(0, steps, steps // 14), [1, steps - 1]]))
    checked = checked[:16]
    kept = torch.empty((checked.shape[0], S, w.d), dtype=torch.int16, device=DEV)
    out = torch.empty((S, w.d), dtype=torch.int16, device=DEV)
    slot = {int(k): j for j, k in enumerate(checked)}
    for k in range(steps):
        scone.scone_decode_step(st, new_d[k], out, rows[k], lens[k])
        if k in slot:
            kept[slot[k]].copy_(out)
    assert scone.scone_status(table) == 0
    rows, lens = rows.cpu().numpy(), lens.cpu().numpy()
    # oracle: Algorithm 1 over prefix ++ new tokens, positions after the prefix
    H = w.K - 1
    seq = np.concatenate([hist, new.T], axis=1)               # [S, H + steps]; hl == H here
    assert (hl == H).all()
    o = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab)
    pos = (np.arange(S)[:, None] * (H + steps) + H + np.arange(steps)[None, :]).reshape(-1)
    o_row, o_len, rc = o.select_at(seq, pos)
    assert rc == 0
    assert np.array_equal(lens.T.reshape(-1), o_len)
    assert np.array_equal(rows.T.reshape(-1), o_row.astype(np.int32))
    assert (o_len == 3).any() and (o_len == 1).any()
    assert checked.shape[0] >= 8
    r = o_row.reshape(S, steps).T[checked]                     # oracle's ids [checked, S]
    t = new[checked]
    exp = np.empty((checked.shape[0], S, w.d), np.uint16)
    hit = r >= 0
    exp[hit] = synth.rows_cpu(synth.F_seed(w), w.d, r[hit])
    exp[~hit] = synth.rows_cpu(synth.T_seed(w), w.d, t[~hit])
    got = kept.cpu().numpy().view(np.uint16)
    bad = np.argwhere((got != exp).any(axis=2))
    assert bad.size == 0, f"{len(bad)} (step, sequence) rows differ, first {bad[0]}"
    st.close()
    table.close()
    buf.free()


def test_prescan_host_mapped_corpus():
    """The training-time pre-scan (Appendix F): scone_match reads a corpus
    held in host memory and writes its tags (row, len) to host memory. Tags
    equal those of the same launch on device copies (where the match walks
    the lengths) and of scone_prescan (staged through HBM), and every
    position equals the oracle."""
    w = synth.WORKLOADS["prescan"].scaled("prescan_test", B=4096)   # 8.4M tokens
    fg_tok, fg_len, _ = synth.fgram_set(w)
    n = w.B * w.L
    F = torch.zeros((w.n_fgrams, w.d), dtype=torch.int16, device=DEV)
    T = torch.zeros((w.vocab, w.d), dtype=torch.int16, device=DEV)
    table = scone.scone_table_build(fg_tok, fg_len, w.K, w.vocab, w.d, F, T)
    corpus = scone.scone_host_alloc(n * 4)
    tags_len = scone.scone_host_alloc(n)
    tags_row = scone.scone_host_alloc(n * 4)
    tok = synth.query_tokens(w, out=corpus.numpy(np.int32)[:n].reshape(w.B, w.L))
    lib = scone.load_library()
    stream = torch.cuda.current_stream().cuda_stream
    assert lib.scone_match(table.handle, corpus.ptr, w.B, w.L, tags_row.ptr, tags_len.ptr,
                           stream) == scone.SCONE_OK
    assert scone.scone_status(table) == 0
    h_len = tags_len.numpy(np.uint8)[:n].copy()
    h_row = tags_row.numpy(np.int32)[:n].copy()
    tok_d = torch.from_numpy(tok).to(DEV)
    row_d = torch.empty(n, dtype=torch.int32, device=DEV)
    ln_d = torch.empty(n, dtype=torch.uint8, device=DEV)
    scone.scone_match(table, tok_d, row_d, ln_d)
    assert np.array_equal(h_len, ln_d.cpu().numpy()) and np.array_equal(h_row, row_d.cpu().numpy())
    o = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab)
    o_row, o_len, _, rc = o.select(tok)
    assert rc == 0
    assert np.array_equal(h_len, o_len.reshape(-1))
    assert np.array_equal(h_row, o_row.reshape(-1).astype(np.int32))
    assert (np.bincount(h_len, minlength=4)[1:] > 0).all()
    # the staged pre-scan (chunks through HBM, eight of them here) writes the same tags
    tags_len.numpy(np.uint8)[:n] = 99
    tags_row.numpy(np.int32)[:n] = -7
    scone.scone_prescan(table, corpus, w.B, w.L, tags_row, tags_len, chunk_tokens=1 << 20)
    assert np.array_equal(tags_len.numpy(np.uint8)[:n], h_len)
    assert np.array_equal(tags_row.numpy(np.int32)[:n], h_row)
    assert scone.scone_status(table) == 0
    table.close()
    for b in (corpus, tags_len, tags_row):
        b.free()


def pack(tok_rows: np.ndarray, lens: np.ndarray) -> np.ndarray:
    """n-grams of tokens < 2^20 (K <= 3) as int64 keys, for membership tests."""
    key = lens.astype(np.int64) << 60
    for j in range(tok_rows.shape[1]):
        t = np.where(j < lens, tok_rows[:, j], 0).astype(np.int64)
        key |= t << (40 - 20 * j)
    return key


def test_fullsize_discover():
    """Algorithm 3 on the 1.07e9-token corpus (K = 3, S = 1e7, count >= 5),
    as the benchmark runs it. Sampled f-grams: counts and first occurrences
    from the oracle's counter; list order; the cut at the threshold. Sampled
    corpus windows: every n-gram above the threshold is selected, none below
    it is."""
    w = synth.WORKLOADS["discover"]
    S = w.n_fgrams
    tok = synth.query_tokens(w)
    tok_d = torch.from_numpy(tok).to(DEV)
    ft, fl, fc, st = scone.scone_fgram_discover(tok_d, w.vocab, w.K, S, w.min_count)
    n = fl.shape[0]
    assert n == S and sum(st["frequent"]) > S           # the cut falls inside the list
    ft, fl, fc = ft.cpu().numpy(), fl.cpu().numpy(), fc.cpu().numpy().astype(np.int64)
    del tok_d
    c_star, at_star = st["threshold"], st["selected_at_threshold"]
    assert (fc >= c_star).all() and (fc >= w.min_count).all()
    assert (fc == c_star).sum() == at_star and (fc > c_star).sum() == S - at_star
    assert np.all(np.diff(fl.astype(np.int64)) >= 0)   # by length
    keys = pack(ft, fl)
    assert np.unique(keys).size == n                   # no n-gram twice
    rng = np.random.default_rng(23)
    # sampled f-grams: exact counts, and first occurrences ascending within a length
    idx = np.sort(rng.choice(n, 3000, replace=False))
    cnt, first = oracle.count_ngrams(tok, w.K, ft[idx], fl[idx])
    assert np.array_equal(cnt, fc[idx]), "counts differ from the oracle's"
    for L_ in (2, 3):
        f = first[fl[idx] == L_]
        assert np.all(np.diff(f) > 0), "not in first-occurrence order"
    # sampled windows: selected iff above the threshold (ties at c* may go either way)
    pos = rng.choice(tok.size, 20000, replace=False)
    flat = tok.reshape(-1)
    q = {}
    for p in pos:
        i = p % w.L
        for m in range(2, w.K + 1):
            if i + 1 >= m:
                q.setdefault(tuple(int(x) for x in flat[p - m + 1:p + 1]), None)
    grams = list(q)
    q_tok = np.full((len(grams), w.K), -1, np.int32)
    q_len = np.array([len(g) for g in grams], np.uint8)
    for k, g in enumerate(grams):
        q_tok[k, :len(g)] = g
    qc, _ = oracle.count_ngrams(tok, w.K, q_tok, q_len)
    chosen = np.isin(pack(q_tok, q_len), keys)
    assert chosen[qc > c_star].all(), "an n-gram above the threshold is missing"
    assert not chosen[(qc < c_star) | (qc < w.min_count)].any(), "an n-gram below it is selected"
    assert chosen.any() and (~chosen).any()
