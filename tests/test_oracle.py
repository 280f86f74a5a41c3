"""The oracle pinned to things other than itself (CPU only).

Pins: the hand-derived K=3 example (tests/golden/hand_k3.json, from
Algorithm 1), brute force over tiny vocabularies, invariants of the
longest-suffix rule on seeded workloads, the K-1 query bound of Sec. 4.3,
special cases that reduce to a library routine (empty V_fgram equals
torch.nn.functional.embedding), and metamorphic relations (permuted f-gram
list, batching, decode equals prefill).
"""

import itertools
import json
import os

import numpy as np
import pytest
import torch

import oracle
import synth
from brute import alg1_sequence

HERE = os.path.dirname(os.path.abspath(__file__))


def marker_rows(n, d, base):
    """Distinct recognisable uint16 rows: row r, column c -> base + 16 r + c."""
    r = np.arange(n, dtype=np.int64)[:, None]
    c = np.arange(d, dtype=np.int64)[None, :]
    return ((base + 16 * r + c) & 0xFFFF).astype(np.uint16)


def pad_fgrams(fgrams, K):
    tok = np.full((len(fgrams), K), -1, np.int32)
    ln = np.zeros(len(fgrams), np.uint8)
    for r, g in enumerate(fgrams):
        tok[r, :len(g)] = g
        ln[r] = len(g)
    return tok, ln


# ------------------------------------------------------------ hand example
def test_hand_example_golden():
    g = json.load(open(os.path.join(HERE, "golden", "hand_k3.json")))
    K, vocab = g["K"], g["vocab"]
    tok = np.array(g["tokens"], np.int32)
    d = 4
    T = marker_rows(vocab, d, 0x1000)
    for case in g["cases"]:
        ft, fl = pad_fgrams(case["fgrams"], K)
        F = marker_rows(len(case["fgrams"]), d, 0x2000)
        o = oracle.Oracle(ft, fl, K, vocab)
        out, row, ln, rc = o.embed(tok, F, T)
        assert rc == 0
        assert row.tolist() == case["row"], case["name"]
        assert ln.tolist() == case["len"], case["name"]
        exp = np.where(np.array(case["row"])[..., None] >= 0,
                       F[np.maximum(np.array(case["row"]), 0)], T[tok])
        assert np.array_equal(out, exp)


def test_hand_example_matches_brute_force():
    g = json.load(open(os.path.join(HERE, "golden", "hand_k3.json")))
    for case in g["cases"]:
        fg = [tuple(x) for x in case["fgrams"]]
        for b, seq in enumerate(g["tokens"]):
            rows, lens = alg1_sequence(seq, fg, g["vocab"])
            assert rows == case["row"][b] and lens == case["len"][b]


# ------------------------------------------------------------- brute force
def _random_case(rng, V, K, p, B, L):
    allg = [g for n in range(2, K + 1) for g in itertools.product(range(V), repeat=n)]
    keep = [g for g in allg if rng.random() < p]
    rng.shuffle(keep)
    tok = rng.integers(0, V, size=(B, L)).astype(np.int32)
    return keep, tok


@pytest.mark.parametrize("V,K", [(2, 2), (2, 3), (3, 3), (2, 5), (3, 5), (4, 5), (4, 3)])
def test_bruteforce_tiny(V, K):
    rng = np.random.default_rng(1000 * V + K)
    for trial in range(12):
        p = [0.0, 0.05, 0.3, 0.7, 1.0][trial % 5]
        L = int(rng.integers(1, 9))
        B = int(rng.integers(1, 4))
        fg, tok = _random_case(rng, V, K, p, B, L)
        ft, fl = pad_fgrams(fg, K)
        o = oracle.Oracle(ft, fl, K, V)
        row, ln, q, rc = o.select(tok)
        assert rc == 0
        for b in range(B):
            rows, lens = alg1_sequence(tok[b].tolist(), fg, V)
            assert row[b].tolist() == rows and ln[b].tolist() == lens, (fg, tok[b])
        assert (q <= K - 1).all()


def test_full_set_gives_longest_possible():
    """V_fgram = all of V^[2,K]: every position takes length min(K, i+1)."""
    V, K = 2, 3
    fg = [g for n in range(2, K + 1) for g in itertools.product(range(V), repeat=n)]
    ft, fl = pad_fgrams(fg, K)
    tok = np.random.default_rng(5).integers(0, V, size=(3, 9)).astype(np.int32)
    row, ln, q, _ = oracle.Oracle(ft, fl, K, V).select(tok)
    exp = np.minimum(K, np.arange(9) + 1)
    assert (ln == exp[None, :]).all()
    # the first scanned query (the longest window) always hits
    assert (q[:, 1:] == 1).all() and (q[:, 0] == 0).all()


def test_all_bigrams_k2():
    """K=2 with every bigram present in the input: len 2 at every i >= 1."""
    tok = np.random.default_rng(7).integers(0, 50, size=(4, 40)).astype(np.int32)
    bigrams = sorted({(int(a), int(b)) for s in tok for a, b in zip(s[:-1], s[1:])})
    ft, fl = pad_fgrams(bigrams, 2)
    row, ln, _, _ = oracle.Oracle(ft, fl, 2, 50).select(tok)
    assert (ln[:, 0] == 1).all() and (ln[:, 1:] == 2).all()
    for b in range(4):
        for i in range(1, 40):
            assert bigrams[row[b, i]] == (tok[b, i - 1], tok[b, i])


# -------------------------------------------------------------- invariants
def check_invariants(fg_tok, fg_len, K, vocab, tok, row, ln, q):
    fset = {tuple(fg_tok[r, :fg_len[r]]) for r in range(len(fg_len))}
    B, L = tok.shape
    for b in range(B):
        s = tok[b]
        for i in range(L):
            r, n = int(row[b, i]), int(ln[b, i])
            top = min(K, i + 1)
            if r >= 0:                                   # 1: selected n-gram is the suffix
                assert 2 <= n <= top
                assert fg_len[r] == n and tuple(fg_tok[r, :n]) == tuple(s[i - n + 1:i + 1])
            else:                                        # 3: fallback <=> no suffix in set
                assert n == 1
            for m in range(max(n + 1, 2), top + 1):      # 2: no longer suffix is in the set
                assert tuple(s[i - m + 1:i + 1]) not in fset
            assert q[b, i] <= K - 1                      # 5: at most K-1 queries (Sec. 4.3)


@pytest.mark.parametrize("name,kw", [
    ("tiny", dict(B=2, L=512)),
    ("stress_k5", dict(B=2, L=1024, quotas=((2, 20000), (3, 20000), (4, 10000), (5, 10000)))),
])
def test_invariants_on_workload(name, kw):
    w = synth.WORKLOADS[name].scaled(name + "_inv", **kw)
    fg_tok, fg_len, _ = synth.fgram_set(w)
    tok = synth.query_tokens(w)
    row, ln, q, rc = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab).select(tok)
    assert rc == 0
    check_invariants(fg_tok, fg_len, w.K, w.vocab, tok, row, ln, q)
    # the workload exercises every length
    for n in range(1, w.K + 1):
        assert (ln == n).any(), n


def test_output_bytes_are_selected_rows():
    """Invariant 4: out equals F[row] or T[token] byte for byte."""
    w = synth.WORKLOADS["tiny"].scaled("tiny_bytes", B=2, L=200, quotas=((2, 2000), (3, 1000)))
    fg_tok, fg_len, _ = synth.fgram_set(w)
    tok = synth.query_tokens(w)
    F = synth.rows_cpu(synth.F_seed(w), w.d, np.arange(w.n_fgrams))
    T = synth.rows_cpu(synth.T_seed(w), w.d, np.arange(w.vocab))
    out, row, ln, rc = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab).embed(tok, F, T)
    assert rc == 0
    exp = np.where(row[..., None] >= 0, F[np.maximum(row, 0)], T[tok])
    assert np.array_equal(out, exp)
    assert (row >= 0).any() and (row < 0).any()


# ----------------------------------------------------------- special cases
def test_empty_set_equals_torch_embedding():
    rng = np.random.default_rng(11)
    V, d = 300, 24
    tok = rng.integers(0, V, size=(3, 50)).astype(np.int32)
    T = rng.integers(0, 2**16, size=(V, d), dtype=np.uint16)
    o = oracle.Oracle(np.zeros((0, 3), np.int32), np.zeros(0, np.uint8), 3, V)
    out, row, ln, rc = o.embed(tok, np.zeros((0, d), np.uint16), T)
    ref = torch.nn.functional.embedding(torch.from_numpy(tok.astype(np.int64)),
                                        torch.from_numpy(T.view(np.int16))).numpy()
    assert rc == 0 and np.array_equal(out.view(np.int16), ref)
    assert (row == -1).all() and (ln == 1).all()


def test_token_out_of_range():
    fg = [(1, 2), (2, 3)]
    ft, fl = pad_fgrams(fg, 3)
    V, d = 5, 4
    tok = np.array([[1, 2, 5, 3, -1, 2, 3], [4, 4, 1, 2, 3, 7, 0]], np.int32)
    T = marker_rows(V, d, 0x1000)
    F = marker_rows(2, d, 0x2000)
    out, row, ln, rc = oracle.Oracle(ft, fl, 3, V).embed(tok, F, T)
    assert rc == oracle.ERR_TOKEN_RANGE
    assert ln.tolist() == [[1, 2, 0, 1, 0, 1, 2], [1, 1, 1, 2, 2, 0, 1]]
    assert row.tolist() == [[-1, 0, -1, -1, -1, -1, 1], [-1, -1, -1, 0, 1, -1, -1]]
    assert (out[0, 2] == 0).all() and (out[0, 4] == 0).all() and (out[1, 5] == 0).all()


def test_rejects_bad_lists():
    ft, fl = pad_fgrams([(1, 2), (3, 4), (1, 2)], 3)
    with pytest.raises(oracle.OracleError) as e:
        oracle.Oracle(ft, fl, 3, 10)
    assert e.value.code == oracle.ERR_DUPLICATE_FGRAM
    ft, fl = pad_fgrams([(1, 2, 3, 4)], 4)
    with pytest.raises(oracle.OracleError):
        oracle.Oracle(ft, fl, 3 + 1, 4)        # token 4 outside vocab 4
    ft = np.array([[1, -1, -1]], np.int32)
    with pytest.raises(oracle.OracleError):
        oracle.Oracle(ft, np.array([1], np.uint8), 3, 10)   # 1-grams are not f-grams


# ------------------------------------------------------------- metamorphic
def _small_workload():
    w = synth.WORKLOADS["tiny"].scaled("tiny_meta", B=3, L=120, quotas=((2, 3000), (3, 2000)))
    fg_tok, fg_len, _ = synth.fgram_set(w)
    tok = synth.query_tokens(w)
    F = synth.rows_cpu(synth.F_seed(w), w.d, np.arange(w.n_fgrams))
    T = synth.rows_cpu(synth.T_seed(w), w.d, np.arange(w.vocab))
    return w, fg_tok, fg_len, tok, F, T


def test_permuted_fgram_list():
    w, fg_tok, fg_len, tok, F, T = _small_workload()
    out, row, ln, _ = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab).embed(tok, F, T)
    perm = np.random.default_rng(3).permutation(w.n_fgrams)
    inv = np.argsort(perm)
    out2, row2, ln2, _ = oracle.Oracle(fg_tok[perm], fg_len[perm], w.K, w.vocab).embed(
        tok, F[perm], T)
    assert np.array_equal(out, out2) and np.array_equal(ln, ln2)
    assert np.array_equal(np.where(row2 >= 0, perm[np.maximum(row2, 0)], -1), row)
    assert np.array_equal(np.where(row >= 0, inv[np.maximum(row, 0)], -1), row2)


def test_batching_equals_single_sequences():
    w, fg_tok, fg_len, tok, F, T = _small_workload()
    o = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab)
    out, row, ln, _ = o.embed(tok, F, T)
    for b in range(tok.shape[0]):
        o1, r1, l1, _ = o.embed(tok[b:b + 1], F, T)
        assert np.array_equal(o1[0], out[b]) and np.array_equal(r1[0], row[b])


def test_select_at_matches_select():
    w, fg_tok, fg_len, tok, F, T = _small_workload()
    o = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab)
    row, ln, _, _ = o.select(tok)
    pos = np.random.default_rng(4).choice(tok.size, 100, replace=False)
    r2, l2, _ = o.select_at(tok, pos)
    assert np.array_equal(r2, row.reshape(-1)[pos]) and np.array_equal(l2, ln.reshape(-1)[pos])


@pytest.mark.parametrize("K", [3, 5])
def test_decode_equals_prefill(K):
    """Embedding token t by decode steps equals prefill on the whole sequence."""
    rng = np.random.default_rng(20 + K)
    V, d, S, steps = 12, 8, 6, 10
    H = K - 1
    full = rng.integers(0, V, size=(S, H + steps)).astype(np.int32)
    # every bigram, so the first step's length always depends on the history,
    # plus longer windows taken from the sequences themselves
    fg = set(itertools.product(range(V), repeat=2))
    for s in range(S):
        for p in range(full.shape[1]):
            n = int(rng.integers(3, K + 1))
            if p + n <= full.shape[1] and rng.random() < 0.3:
                fg.add(tuple(full[s, p:p + n].tolist()))
    fg = sorted(fg)
    ft, fl = pad_fgrams(fg, K)
    o = oracle.Oracle(ft, fl, K, V)
    F = marker_rows(len(fg), d, 0x2000)
    T = marker_rows(V, d, 0x1000)
    hl = np.array([0, 1, H, H, 2 if H >= 2 else 1, 1], np.int32)[:S]
    # entries left of the last hist_len ones must be ignored: fill them with valid tokens
    hist = rng.integers(0, V, size=(S, H)).astype(np.int32)
    for s in range(S):
        if hl[s]:
            hist[s, H - hl[s]:] = full[s, H - hl[s]:H]
    new = np.ascontiguousarray(full[:, H:].T)
    out, row, ln, rc = o.decode(hist, hl, new, F, T)
    assert rc == 0
    for s in range(S):
        seq = full[s, H - hl[s]:][None, :]
        po, pr, pl, _ = o.embed(seq, F, T)
        h = int(hl[s])
        assert np.array_equal(out[:, s], po[0, h:])
        assert np.array_equal(row[:, s], pr[0, h:]) and np.array_equal(ln[:, s], pl[0, h:])
        assert (ln[:, s] >= 2).sum() >= steps - 1
    assert (ln[0, hl > 0] >= 2).all() and (ln[0, hl == 0] == 1).all()
    assert (ln > 2).any()


@pytest.mark.parametrize("threads", [2, 5, 64])
def test_threaded_embed_equals_single_thread(threads):
    """The std::thread split over sequences (used for the multi-core CPU
    timing) gives the single-thread result, including the status of an
    out-of-range token in one of the ranges."""
    w = synth.WORKLOADS["tiny"].scaled("tiny_mt", B=9, L=37)
    ft, fl, _ = synth.fgram_set(w)
    tok = synth.query_tokens(w)
    tok[6, 11] = w.vocab
    F = synth.rows_cpu(synth.F_seed(w), w.d, np.arange(len(fl)))
    T = synth.rows_cpu(synth.T_seed(w), w.d, np.arange(w.vocab))
    o = oracle.Oracle(ft, fl, w.K, w.vocab)
    a = o.embed(tok, F, T)
    b = o.embed(tok, F, T, threads=threads)
    assert a[3] == b[3] == oracle.ERR_TOKEN_RANGE
    for x, y in zip(a[:3], b[:3]):
        assert np.array_equal(x, y)
