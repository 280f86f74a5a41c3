"""The f-gram discovery oracle (Algorithm 3) pinned to things other than
itself (CPU only).

Pins: the hand-derived example (tests/golden/hand_discover.json), the literal
algorithm by brute force over tiny vocabularies (every n-gram of the
vocabulary counted against every window), closed forms (a repeated token, an
alternating pair, all-distinct tokens, the sequence boundary), and invariants
on seeded Zipf corpora (window totals, counts never grow with length, the
top-S cut, the query-map counter agreeing with the full count map).
"""

import itertools
import json
import os

import numpy as np
import pytest

import oracle
import synth
from brute import alg3_counts, alg3_select

HERE = os.path.dirname(os.path.abspath(__file__))


def as_list(res):
    return [tuple(int(x) for x in t[:n]) for t, n in zip(res["tok"], res["len"])]


def test_hand_example():
    g = json.load(open(os.path.join(HERE, "golden", "hand_discover.json")))
    tok = np.array(g["tokens"], np.int32)
    K, V = g["K"], g["vocab"]
    full = oracle.discover(tok, K, V, 1000, 1)
    want = {tuple(w): (c, f) for w, c, f in zip(g["counts"]["grams"], g["counts"]["count"],
                                                 g["counts"]["first"])}
    got = dict(zip(as_list(full), (int(c) for c in full["count"])))
    assert got == {w: c for w, (c, _) in want.items()}
    assert list(full["distinct"]) == g["counts"]["distinct"]
    assert list(oracle.discover(tok, K, V, 1000, 2)["frequent"]) == g["counts"]["frequent_at_2"]
    for case in g["cases"]:
        r = oracle.discover(tok, K, V, case["S"], case["min_count"])
        assert as_list(r) == [tuple(w) for w in case["grams"]], case["why"]
        assert list(r["count"]) == case["count"], case["why"]
        assert r["tok"].shape[1] == K and all((t[n:] == -1).all() for t, n in zip(r["tok"], r["len"]))


@pytest.mark.parametrize("V,K", [(2, 2), (2, 4), (3, 3), (4, 2)])
def test_brute_force_tiny(V, K):
    rng = np.random.default_rng(100 * V + K)
    for trial in range(12):
        B = int(rng.integers(1, 4))
        L = int(rng.integers(0, 9))
        tok = rng.integers(0, V, size=(B, L)).astype(np.int32)
        counts = alg3_counts(tok.tolist(), V, K)
        for S, mc in itertools.product((0, 1, 3, 7, 1000), (1, 2, 3)):
            r = oracle.discover(tok, K, V, S, mc)
            sel = alg3_select(counts, S, mc)
            assert as_list(r) == [w for w, _, _ in sel], (tok.tolist(), S, mc)
            assert list(r["count"]) == [c for _, c, _ in sel]
        r = oracle.discover(tok, K, V, 10 ** 6, 1)
        for n in range(2, K + 1):
            assert r["distinct"][n] == sum(1 for w in counts if len(w) == n)


def test_repeated_token():
    """One sequence x^L: the n-gram x^n appears L - n + 1 times."""
    for L, K in [(1, 3), (2, 3), (7, 3), (9, 5), (3, 8)]:
        tok = np.full((1, L), 4, np.int32)
        r = oracle.discover(tok, K, 5, 100, 1)
        ns = [n for n in range(2, K + 1) if n <= L]
        assert as_list(r) == [(4,) * n for n in ns]
        assert list(r["count"]) == [L - n + 1 for n in ns]


def test_alternating_pair():
    """(a b)^m: ab appears m times, ba m - 1, aba and bab m - 1 each."""
    m = 6
    tok = np.array([[3, 1] * m], np.int32)
    r = oracle.discover(tok, 3, 4, 100, 1)
    assert as_list(r) == [(3, 1), (1, 3), (3, 1, 3), (1, 3, 1)]
    assert list(r["count"]) == [m, m - 1, m - 1, m - 1]
    r = oracle.discover(tok, 3, 4, 1, 1)
    assert as_list(r) == [(3, 1)]
    # the three grams tied at m - 1: the bigram first, then aba by first occurrence
    r = oracle.discover(tok, 3, 4, 3, 1)
    assert as_list(r) == [(3, 1), (1, 3), (3, 1, 3)]


def test_all_distinct_tokens():
    """Every window is a different n-gram: count 1 each, listed in corpus order."""
    L, K = 12, 4
    tok = np.arange(2 * L, dtype=np.int32).reshape(2, L)
    assert as_list(oracle.discover(tok, K, 2 * L, 10 ** 6, 2)) == []
    r = oracle.discover(tok, K, 2 * L, 10 ** 6, 1)
    want = [tuple(int(x) for x in tok[b, p:p + n]) for n in range(2, K + 1)
            for b in range(2) for p in range(L - n + 1)]
    assert as_list(r) == want
    assert (r["count"] == 1).all()
    # S cuts inside the bigrams, by first occurrence
    assert as_list(oracle.discover(tok, K, 2 * L, 5, 1)) == want[:5]


def test_sequence_boundary():
    r = oracle.discover(np.array([[1, 2], [3, 4]], np.int32), 3, 5, 100, 1)
    assert as_list(r) == [(1, 2), (3, 4)]


def test_errors():
    tok = np.array([[1, 2, 3]], np.int32)
    for args in [(1, 5, 10, 1), (9, 5, 10, 1), (3, 5, -1, 1), (3, 5, 10, 0)]:
        with pytest.raises(oracle.OracleError) as e:
            oracle.discover(tok, *args)
        assert e.value.code == oracle.ERR_INVALID_ARG
    with pytest.raises(oracle.OracleError) as e:
        oracle.discover(tok, 3, 3, 10, 1)           # token 3 outside [0, 3)
    assert e.value.code == oracle.ERR_TOKEN_RANGE
    with pytest.raises(oracle.OracleError) as e:
        oracle.discover(np.array([[1, -1]], np.int32), 3, 5, 10, 1)
    assert e.value.code == oracle.ERR_TOKEN_RANGE
    r = oracle.discover(np.zeros((0, 5), np.int32), 3, 5, 10, 1)
    assert r["len"].size == 0


def zipf_corpus(B, L, V, seed):
    w = synth.WORKLOADS["tiny"].scaled("discover_pin", B=B, L=L, vocab=V)
    return synth.zipf_tokens(w, seed, B * L, inject=False).reshape(B, L)


@pytest.mark.parametrize("K,mc", [(3, 1), (4, 2), (5, 5)])
def test_invariants_zipf(K, mc):
    B, L, V = 6, 400, 300
    tok = zipf_corpus(B, L, V, seed=K)
    full = oracle.discover(tok, K, V, 10 ** 7, 1)
    grams = as_list(full)
    count = dict(zip(grams, (int(c) for c in full["count"])))
    # every window is counted once
    for n in range(2, K + 1):
        assert sum(c for g, c in count.items() if len(g) == n) == B * (L - n + 1)
    # a gram never appears more often than its prefix or its suffix
    for g, c in count.items():
        if len(g) > 2:
            assert c <= count[g[:-1]] and c <= count[g[1:]]
    # the threshold keeps exactly the grams at or above it
    freq = oracle.discover(tok, K, V, 10 ** 7, mc)
    assert set(as_list(freq)) == {g for g, c in count.items() if c >= mc}
    for n in range(2, K + 1):
        assert freq["frequent"][n] == sum(1 for g, c in count.items() if len(g) == n and c >= mc)
    # top-S: nothing left out is more frequent than anything selected
    S = len(freq["len"]) // 3
    top = oracle.discover(tok, K, V, S, mc)
    assert len(top["len"]) == S
    chosen = set(as_list(top))
    rest = [count[g] for g in count if g not in chosen and count[g] >= mc]
    assert min(top["count"]) >= max(rest)
    # the query-map counter agrees with the full count map, first occurrences included
    sample = np.random.default_rng(K).choice(len(grams), 200, replace=False)
    q_tok = full["tok"][sample]
    q_len = full["len"][sample]
    c, first = oracle.count_ngrams(tok, K, q_tok, q_len)
    assert list(c) == [count[grams[i]] for i in sample]
    flat = tok.reshape(-1)
    for qi, f in zip(sample, first):
        n = len(grams[qi])
        assert tuple(int(x) for x in flat[f:f + n]) == grams[qi]


def test_count_ngrams_brute():
    rng = np.random.default_rng(7)
    tok = rng.integers(0, 3, size=(3, 7)).astype(np.int32)
    counts = alg3_counts(tok.tolist(), 3, 4)
    absent = [g for g in [(2, 2, 2, 2), (0, 1, 0, 1), (1, 1)] if g not in counts]
    assert absent
    grams = list(counts) + absent
    q_tok = np.full((len(grams), 4), -1, np.int32)
    q_len = np.array([len(g) for g in grams], np.uint8)
    for i, g in enumerate(grams):
        q_tok[i, :len(g)] = g
    c, first = oracle.count_ngrams(tok, 4, q_tok, q_len)
    for i, g in enumerate(grams):
        want = counts.get(g, (0, -1))
        assert (int(c[i]), int(first[i])) == want, g
