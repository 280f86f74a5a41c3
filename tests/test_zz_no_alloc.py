"""scone_table_rebuild_noalloc: swapping f-gram lists without allocating (GPU).

Some callers may not allocate when they swap in a new f-gram list: a serving
process whose device memory is owned by another allocator (cudaMalloc would
fail or fragment it), or a latency-bound thread that must not pay for
cudaMalloc / cudaFree, which can synchronize the whole device. For them the
library offers one entry point that reuses the table's own memory and keeps
the build kernels' scratch in a fixed device array. Its tables must behave
exactly like tables from scone_table_build, call after call, although every
call reuses the same scratch.

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes when run on its own.
"""

import ctypes

import numpy as np
import pytest
import torch

import synth
import paper_2502_01637_gb300 as scone
from gpu_cases import DEV, dev_rows, run_embed

pytestmark = pytest.mark.gpu

BASE = synth.WORKLOADS["tiny"].scaled("noalloc_a", B=3, L=400,
                                      quotas=((2, 30000), (3, 20000)))
OTHER = synth.Workload("noalloc_b", 77, BASE.vocab, BASE.zipf_s, BASE.B, BASE.L,
                       ((2, 20000), (3, 25000)), BASE.K, BASE.d)


def _rows(w, n):
    return dev_rows(synth.rows_cpu(synth.F_seed(w), w.d, np.arange(n)))


def _rebuild_via_c_abi(table, fg_tok, fg_len, F):
    """Calls the C entry point directly (the ctypes signature is the header's)."""
    lib = scone.load_library()
    ft = np.ascontiguousarray(fg_tok, np.int32)
    fl = np.ascontiguousarray(fg_len, np.uint8)
    n = fl.shape[0]
    return lib.scone_table_rebuild_noalloc(table.handle, ft.ctypes.data if n else None,
                                           fl.ctypes.data if n else None, n,
                                           F.data_ptr() if n else None,
                                           torch.cuda.current_stream().cuda_stream)


def _same_as_fresh_build(table, fg_tok, fg_len, F, T, tok):
    ref = scone.scone_table_build(fg_tok, fg_len, BASE.K, BASE.vocab, BASE.d, F, T)
    a = run_embed(table, tok, BASE.d)
    b = run_embed(ref, tok, BASE.d)
    ref.close()
    # bit-exact, the tolerance every parity test of this path uses
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    return a


def test_rebuild_noalloc_matches_build_on_two_calls_in_a_row():
    fg1_tok, fg1_len, _ = synth.fgram_set(BASE)
    fg2_tok, fg2_len, _ = synth.fgram_set(OTHER)
    T = dev_rows(synth.rows_cpu(synth.T_seed(BASE), BASE.d, np.arange(BASE.vocab)))
    F1 = _rows(BASE, BASE.n_fgrams)
    F2 = _rows(OTHER, OTHER.n_fgrams)
    tok = synth.query_tokens(BASE)
    table = scone.scone_table_build(fg1_tok, fg1_len, BASE.K, BASE.vocab, BASE.d, F1, T)
    assert OTHER.n_fgrams <= 0.85 * table.info()["n_slots"]
    # two calls in a row, each compared with a table built the ordinary way
    for fg_tok, fg_len, F in ((fg2_tok, fg2_len, F2), (fg1_tok, fg1_len, F1)):
        assert _rebuild_via_c_abi(table, fg_tok, fg_len, F) == scone.SCONE_OK
        out, row, ln = _same_as_fresh_build(table, fg_tok, fg_len, F, T, tok)
        assert table.info()["n_fgrams"] == fg_len.shape[0]
        assert (ln >= 2).any() and (ln == 1).any()
    assert scone.scone_status(table) == scone.SCONE_OK
    table.close()


def test_rebuild_noalloc_clears_its_flags_and_rejects_oversize_lists():
    fg_tok, fg_len, _ = synth.fgram_set(BASE)
    T = dev_rows(synth.rows_cpu(synth.T_seed(BASE), BASE.d, np.arange(BASE.vocab)))
    F = _rows(BASE, BASE.n_fgrams)
    tok = synth.query_tokens(BASE)
    table = scone.scone_table_build(fg_tok, fg_len, BASE.K, BASE.vocab, BASE.d, F, T)
    # a list holding a duplicate: reported, and the table is left empty (all T)
    dup_tok = np.concatenate([fg_tok[:100], fg_tok[:1]])
    dup_len = np.concatenate([fg_len[:100], fg_len[:1]])
    assert _rebuild_via_c_abi(table, dup_tok, dup_len, F) == scone.SCONE_ERR_DUPLICATE_FGRAM
    out, row, ln = run_embed(table, tok, BASE.d)
    assert (row == -1).all() and (ln == 1).all()
    # the next call starts from cleared flags and succeeds
    assert _rebuild_via_c_abi(table, fg_tok, fg_len, F) == scone.SCONE_OK
    _same_as_fresh_build(table, fg_tok, fg_len, F, T, tok)
    # more f-grams than 0.85 of the slots: refused before any device work
    n_slots = table.info()["n_slots"]
    big = int(0.85 * n_slots) + 1
    big_tok = np.zeros((big, BASE.K), np.int32)
    big_len = np.full(big, 2, np.uint8)
    assert _rebuild_via_c_abi(table, big_tok, big_len, F) == scone.SCONE_ERR_INVALID_ARG
    # the table is untouched by the refused call
    _same_as_fresh_build(table, fg_tok, fg_len, F, T, tok)
    table.close()


def _distinct_trigrams(n, vocab):
    i = np.arange(n, dtype=np.int64)
    tok = np.stack([i // (vocab * vocab), (i // vocab) % vocab, i % vocab], 1).astype(np.int32)
    return tok, np.full(n, 3, np.uint8)


def test_rebuild_noalloc_scratch_limit():
    """Lists up to the fixed scratch work; one past it is refused with a clear
    error before any device work, and the table keeps its previous list."""
    K, vocab, d = 3, 1000, 8
    scratch = 16 << 20                                  # SCONE_REBUILD_SCRATCH_BYTES
    n_under, n_over = 1_200_000, 1_300_000
    need = lambda n: 256 + -(-n // 256) * 256 + -(-(n * 4 * K) // 256) * 256
    assert need(n_under) <= scratch < need(n_over)
    T = dev_rows(np.zeros((vocab, d), np.uint16))
    ft0, fl0 = _distinct_trigrams(100_000, vocab)
    F = dev_rows(np.arange(n_over * d, dtype=np.uint16).reshape(n_over, d))
    table = scone.scone_table_build(ft0, fl0, K, vocab, d, F[:100_000], T, load_factor=0.05)
    assert n_over <= 0.85 * table.info()["n_slots"]     # only the scratch limit applies
    ft, fl = _distinct_trigrams(n_under, vocab)
    assert _rebuild_via_c_abi(table, ft, fl, F) == scone.SCONE_OK
    tok = ft[::997][:, :].reshape(-1)[None, :]          # windows that hit many f-grams
    ref = scone.scone_table_build(ft, fl, K, vocab, d, F[:n_under], T)
    a, b = run_embed(table, tok, d), run_embed(ref, tok, d)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    assert (a[2] == 3).any()
    ref.close()
    ft2, fl2 = _distinct_trigrams(n_over, vocab)
    assert _rebuild_via_c_abi(table, ft2, fl2, F) == scone.SCONE_ERR_INVALID_ARG
    assert table.info()["n_fgrams"] == n_under
    c = run_embed(table, tok, d)
    for x, y in zip(a, c):
        assert np.array_equal(x, y)
    table.close()
