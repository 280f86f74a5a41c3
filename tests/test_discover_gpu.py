"""f-gram discovery on the GPU (Algorithm 3 by the K-1 counting scans of
Sec. 3.2) against the oracle, which counts every n-gram in a map without
pruning (GPU).

Small corpora: the whole list (tokens, lengths, counts) and the per-length
statistics are compared exactly, over lengths K = 2..8, thresholds 1..5 and
cuts S below, at and above the number of eligible n-grams, at sizes spanning
several aggregation chunks with a ragged tail. Edge cases: empty and
one-token sequences, sequences shorter than K, a single repeated token, an
out-of-range token. The discovered list then drives the embedding path end
to end.
"""

import json
import os

import numpy as np
import pytest
import torch

import oracle
import synth
import paper_2502_01637_gb300 as scone
from gpu_cases import DEV, SmallCase

pytestmark = pytest.mark.gpu
HERE = os.path.dirname(os.path.abspath(__file__))


def gpu_discover(tok, vocab, K, S, mc):
    t = torch.from_numpy(np.ascontiguousarray(tok, np.int32)).to(DEV)
    ft, fl, fc, st = scone.scone_fgram_discover(t, vocab, K, S, mc)
    torch.cuda.synchronize()
    return ft.cpu().numpy(), fl.cpu().numpy(), fc.cpu().numpy().view(np.uint32), st


def assert_same(tok, vocab, K, S, mc):
    ref = oracle.discover(tok, K, vocab, S, mc)
    ft, fl, fc, st = gpu_discover(tok, vocab, K, S, mc)
    assert np.array_equal(fl, ref["len"]), (K, S, mc)
    assert np.array_equal(ft, ref["tok"]), (K, S, mc)
    assert np.array_equal(fc, ref["count"]), (K, S, mc)
    for n in range(2, K + 1):
        assert st["frequent"][n] == ref["frequent"][n], ("frequent", n, K, mc)
    assert st["distinct"][2] == ref["distinct"][2]
    if mc == 1:   # nothing is pruned: every length sees every window
        for n in range(2, K + 1):
            assert st["distinct"][n] == ref["distinct"][n]
    return ref, st


def test_hand_example():
    g = json.load(open(os.path.join(HERE, "golden", "hand_discover.json")))
    tok = np.array(g["tokens"], np.int32)
    for case in g["cases"]:
        ft, fl, fc, _ = gpu_discover(tok, g["vocab"], g["K"], case["S"], case["min_count"])
        got = [tuple(int(x) for x in t[:n]) for t, n in zip(ft, fl)]
        assert got == [tuple(w) for w in case["grams"]], case["why"]
        assert list(fc) == case["count"], case["why"]


def zipf(B, L, V, seed, s=1.1):
    w = synth.WORKLOADS["tiny"].scaled("disc_gpu", B=B, L=L, vocab=V, zipf_s=s)
    return synth.zipf_tokens(w, seed, B * L, inject=False).reshape(B, L)


@pytest.mark.parametrize("K", [2, 3, 4, 5, 8])
@pytest.mark.parametrize("mc", [1, 2, 5])
def test_small_corpora(K, mc):
    # 3 x 1500: two 2048-window aggregation chunks and a ragged third
    tok = zipf(3, 1500, 40, seed=K * 10 + mc)
    full = oracle.discover(tok, K, 40, 10 ** 7, mc)
    M = len(full["len"])
    assert M > 10
    for S in sorted({0, 1, 7, M // 2, M - 1, M, M + 10}):
        assert_same(tok, 40, K, S, mc)


def test_many_chunks_and_hot_keys():
    """64 x 700 tokens of a 12-token vocabulary: every chunk repeats its keys
    hundreds of times, and keys recur across 22 chunks."""
    tok = zipf(64, 700, 12, seed=3)
    for K, mc, S in [(3, 1, 50), (4, 5, 300), (6, 2, 10 ** 6)]:
        assert_same(tok, 12, K, S, mc)


def test_larger_vocab_multiscan():
    tok = zipf(32, 4096, 2000, seed=11)
    ref = oracle.discover(tok, 4, 2000, 10 ** 7, 3)
    M = len(ref["len"])
    for S in (M // 3, M):
        assert_same(tok, 2000, 4, S, 3)


def test_edge_shapes():
    rng = np.random.default_rng(1)
    for B, L, K in [(5, 1, 3), (4, 2, 3), (3, 3, 5), (1, 7, 8), (2, 0, 3)]:
        tok = rng.integers(0, 3, size=(B, L)).astype(np.int32)
        assert_same(tok, 3, K, 100, 1)
    tok = np.full((2, 3000), 6, np.int32)     # one key per length, hot in every chunk
    ref, _ = assert_same(tok, 7, 5, 10, 1)
    assert list(ref["count"]) == [2 * (3000 - n + 1) for n in range(2, 6)]
    ft, fl, fc, st = gpu_discover(np.zeros((0, 16), np.int32), 5, 3, 10, 1)
    assert fl.size == 0


def test_token_range_error():
    tok = zipf(2, 500, 30, seed=2)
    tok[1, 17] = 30
    t = torch.from_numpy(tok).to(DEV)
    with pytest.raises(scone.SconeError) as e:
        scone.scone_fgram_discover(t, 30, 3, 100, 1)
    assert e.value.code == scone.SCONE_ERR_TOKEN_RANGE
    tok[1, 17] = -4
    t = torch.from_numpy(tok).to(DEV)
    with pytest.raises(scone.SconeError) as e:
        scone.scone_fgram_discover(t, 30, 3, 100, 1)
    assert e.value.code == scone.SCONE_ERR_TOKEN_RANGE


def test_discovered_set_drives_embedding():
    """Corpus -> discovered f-grams -> table -> Algorithm 1, against the
    oracle run on the oracle's own discovered list."""
    w = synth.WORKLOADS["tiny"].scaled("disc_e2e", B=4, L=600, vocab=500, d=64)
    corpus = zipf(16, 2048, 500, seed=9)
    ref = oracle.discover(corpus, 3, 500, 4000, 5)
    ft, fl, fc, _ = gpu_discover(corpus, 500, 3, 4000, 5)
    assert np.array_equal(ft, ref["tok"]) and np.array_equal(fl, ref["len"])
    case = SmallCase(w, fgrams=(ft, fl), tok=zipf(4, 600, 500, seed=10))
    table = case.build()
    out_exp, row_exp, len_exp, rc = case.expected()
    assert rc == 0
    t = torch.from_numpy(case.tok).to(DEV)
    out = torch.empty((t.numel(), w.d), dtype=torch.int16, device=DEV)
    row = torch.empty(t.numel(), dtype=torch.int32, device=DEV)
    ln = torch.empty(t.numel(), dtype=torch.uint8, device=DEV)
    scone.scone_embed(table, t, out, row, ln)
    scone.scone_status(table)
    assert np.array_equal(row.cpu().numpy(), row_exp.reshape(-1).astype(np.int32))
    assert np.array_equal(ln.cpu().numpy(), len_exp.reshape(-1))
    assert np.array_equal(out.cpu().numpy().view(np.uint16), out_exp.reshape(-1, w.d))
    assert (ln.cpu().numpy() == 3).any()
    table.close()


def test_workspace_reuse():
    """A workspace reused across corpora (growing, then smaller) gives the
    results of calls without one; its buffers stay allocated."""
    ws = scone.scone_discover_create()
    for B, L, V, K, mc in [(2, 900, 30, 3, 2), (8, 3000, 60, 4, 3), (3, 500, 20, 5, 1)]:
        tok = zipf(B, L, V, seed=B + L)
        t = torch.from_numpy(tok).to(DEV)
        a = scone.scone_fgram_discover(t, V, K, 500, mc, workspace=ws)
        b = scone.scone_fgram_discover(t, V, K, 500, mc)
        for x, y in zip(a[:3], b[:3]):
            assert torch.equal(x, y)
        assert a[3]["workspace_bytes"] > 0 and b[3]["frequent"] == a[3]["frequent"]
        ref = oracle.discover(tok, K, V, 500, mc)
        assert np.array_equal(a[1].cpu().numpy(), ref["len"])
        assert np.array_equal(a[0].cpu().numpy(), ref["tok"])
    ws.close()


@pytest.mark.parametrize("slack", [0.02, 0.5, 4.0, 40.0])
def test_table_sizing_and_rebuild(slack):
    """The counting table is sized from a sketch of the distinct n-grams;
    the sizing never changes the result. A table far too small for the keys
    fills up and the scan is counted again in a worst-case table; at the
    default and above nothing is rebuilt, and the sketch stays within a few
    percent of the exact distinct count."""
    V, K, mc = 3000, 4, 2
    tok = zipf(16, 4000, V, seed=11)
    ws = scone.scone_discover_create()
    ws.set_table_slack(slack)
    t = torch.from_numpy(tok).to(DEV)
    ft, fl, fc, st = scone.scone_fgram_discover(t, V, K, 5000, mc, workspace=ws)
    ref = oracle.discover(tok, K, V, 5000, mc)
    assert np.array_equal(fl.cpu().numpy(), ref["len"])
    assert np.array_equal(ft.cpu().numpy(), ref["tok"])
    assert np.array_equal(fc.cpu().numpy().view(np.uint32), ref["count"])
    for n in range(2, K + 1):
        assert st["frequent"][n] == ref["frequent"][n]
        assert abs(st["estimate"][n] - st["distinct"][n]) <= 0.06 * st["distinct"][n] + 8, n
    if slack < 1:
        assert st["table_rebuilds"] >= 1
    else:
        assert st["table_rebuilds"] == 0
    ws.close()
