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

import numpy as np
import pytest
import torch

import oracle
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


def _same_as_oracle(got, fg_tok, fg_len, F_host, T_host, tok, K=BASE.K, vocab=BASE.vocab):
    """Element-wise equality of (out, row, len) with the oracle of Algorithm 1."""
    o_out, o_row, o_len, rc = oracle.Oracle(fg_tok, fg_len, K, vocab).embed(tok, F_host, T_host)
    assert rc == oracle.OK
    out, row, ln = got
    assert np.array_equal(row, o_row.reshape(-1).astype(np.int32))
    assert np.array_equal(ln, o_len.reshape(-1))
    assert np.array_equal(out, o_out.reshape(out.shape))


def _no_alloc_call(table, fg_tok, fg_len, F):
    """One call with the device's free memory and torch's allocation counters
    read on both sides: neither may move."""
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    n0 = torch.cuda.memory_stats().get("allocation.all.allocated", 0)
    rc = _rebuild_via_c_abi(table, fg_tok, fg_len, F)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    n1 = torch.cuda.memory_stats().get("allocation.all.allocated", 0)
    assert free1 == free0, f"device free memory moved by {free0 - free1} bytes"
    assert n1 == n0
    return rc


def test_rebuild_noalloc_matches_build_on_two_calls_in_a_row():
    fg1_tok, fg1_len, _ = synth.fgram_set(BASE)
    fg2_tok, fg2_len, _ = synth.fgram_set(OTHER)
    T_host = synth.rows_cpu(synth.T_seed(BASE), BASE.d, np.arange(BASE.vocab))
    F1_host = synth.rows_cpu(synth.F_seed(BASE), BASE.d, np.arange(BASE.n_fgrams))
    F2_host = synth.rows_cpu(synth.F_seed(OTHER), OTHER.d, np.arange(OTHER.n_fgrams))
    T, F1, F2 = dev_rows(T_host), dev_rows(F1_host), dev_rows(F2_host)
    tok = synth.query_tokens(BASE)
    table = scone.scone_table_build(fg1_tok, fg1_len, BASE.K, BASE.vocab, BASE.d, F1, T)
    assert OTHER.n_fgrams <= 0.85 * table.info()["n_slots"]
    # two calls in a row, each compared with a table built the ordinary way
    # and with the oracle; the second call must not move the device's free
    # memory (the first may load the library's module on a fresh device)
    calls = ((fg2_tok, fg2_len, F2, F2_host), (fg1_tok, fg1_len, F1, F1_host))
    for k, (fg_tok, fg_len, F, F_host) in enumerate(calls):
        if k == 0:
            assert _rebuild_via_c_abi(table, fg_tok, fg_len, F) == scone.SCONE_OK
        else:
            assert _no_alloc_call(table, fg_tok, fg_len, F) == scone.SCONE_OK
        got = _same_as_fresh_build(table, fg_tok, fg_len, F, T, tok)
        _same_as_oracle(got, fg_tok, fg_len, F_host, T_host, tok)
        assert table.info()["n_fgrams"] == fg_len.shape[0]
        assert (got[2] >= 2).any() and (got[2] == 1).any()
    assert scone.scone_status(table) == scone.SCONE_OK
    table.close()


def test_rebuild_noalloc_host_mapped_F():
    """F in pinned, device-mapped host memory (the offloaded tier): the new
    list's rows are read through the mapped address of the new buffer."""
    fg1_tok, fg1_len, _ = synth.fgram_set(BASE)
    fg2_tok, fg2_len, _ = synth.fgram_set(OTHER)
    T_host = synth.rows_cpu(synth.T_seed(BASE), BASE.d, np.arange(BASE.vocab))
    T = dev_rows(T_host)
    tok = synth.query_tokens(BASE)
    bufs, hosts = [], []
    for w in (BASE, OTHER):
        h = synth.rows_cpu(synth.F_seed(w), w.d, np.arange(w.n_fgrams))
        b = scone.scone_host_alloc(h.nbytes)
        b.numpy(np.uint16)[:h.size] = h.reshape(-1)
        bufs.append(b)
        hosts.append(h)
    table = scone.scone_table_build(fg1_tok, fg1_len, BASE.K, BASE.vocab, BASE.d, bufs[0].ptr,
                                    T, F_location=scone.SCONE_ROWS_HOST_MAPPED)
    calls = ((fg2_tok, fg2_len, bufs[1], hosts[1]), (fg1_tok, fg1_len, bufs[0], hosts[0]))
    for fg_tok, fg_len, b, h in calls:
        lib = scone.load_library()
        rc = lib.scone_table_rebuild_noalloc(
            table.handle, np.ascontiguousarray(fg_tok, np.int32).ctypes.data,
            np.ascontiguousarray(fg_len, np.uint8).ctypes.data, fg_len.shape[0], b.ptr,
            torch.cuda.current_stream().cuda_stream)
        assert rc == scone.SCONE_OK
        assert table.info()["F_location"] == scone.SCONE_ROWS_HOST_MAPPED
        _same_as_oracle(run_embed(table, tok, BASE.d), fg_tok, fg_len, h, T_host, tok)
    assert scone.scone_status(table) == scone.SCONE_OK
    table.close()
    for b in bufs:
        b.free()


def test_wrapper_keeps_the_old_F_after_a_refused_call():
    """A refused call leaves the table on its old list and old F; the Python
    wrapper must keep that F alive even when the caller drops it."""
    fg_tok, fg_len, _ = synth.fgram_set(BASE)
    T_host = synth.rows_cpu(synth.T_seed(BASE), BASE.d, np.arange(BASE.vocab))
    F_host = synth.rows_cpu(synth.F_seed(BASE), BASE.d, np.arange(BASE.n_fgrams))
    T, F = dev_rows(T_host), dev_rows(F_host)
    tok = synth.query_tokens(BASE)
    table = scone.scone_table_build(fg_tok, fg_len, BASE.K, BASE.vocab, BASE.d, F, T)
    n_slots = table.info()["n_slots"]
    big = int(0.85 * n_slots) + 1
    F_big = torch.zeros((big, BASE.d), dtype=torch.int16, device=DEV)
    with pytest.raises(scone.SconeError) as e:
        scone.scone_table_rebuild_noalloc(table, np.zeros((big, BASE.K), np.int32),
                                          np.full(big, 2, np.uint8), F_big)
    assert e.value.code == scone.SCONE_ERR_INVALID_ARG
    # drop the caller's references; a same-sized allocation would take the old
    # F's block from torch's cache if the wrapper had released it
    nbytes = F.numel()
    del F, F_big
    junk = torch.full((nbytes,), -1, dtype=torch.int16, device=DEV)
    _same_as_oracle(run_embed(table, tok, BASE.d), fg_tok, fg_len, F_host, T_host, tok)
    del junk
    table.close()


def test_graphs_captured_again_after_a_rebuild():
    """A graph captured before the call keeps the old list's state; captured
    again after it, it gives the new list's result, bit for bit."""
    fg1_tok, fg1_len, _ = synth.fgram_set(BASE)
    fg2_tok, fg2_len, _ = synth.fgram_set(OTHER)
    T_host = synth.rows_cpu(synth.T_seed(BASE), BASE.d, np.arange(BASE.vocab))
    F1_host = synth.rows_cpu(synth.F_seed(BASE), BASE.d, np.arange(BASE.n_fgrams))
    F2_host = synth.rows_cpu(synth.F_seed(OTHER), OTHER.d, np.arange(OTHER.n_fgrams))
    T, F1, F2 = dev_rows(T_host), dev_rows(F1_host), dev_rows(F2_host)
    tok = synth.query_tokens(BASE)
    tok_d = torch.from_numpy(tok).to(DEV)
    n = tok.size
    out = torch.empty((n, BASE.d), dtype=torch.int16, device=DEV)
    row = torch.empty(n, dtype=torch.int32, device=DEV)
    ln = torch.empty(n, dtype=torch.uint8, device=DEV)
    table = scone.scone_table_build(fg1_tok, fg1_len, BASE.K, BASE.vocab, BASE.d, F1, T)

    def capture():
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            scone.scone_embed(table, tok_d, out, row, ln)      # warm-up outside capture
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            scone.scone_embed(table, tok_d, out, row, ln)
        return g

    def replay(g):
        out.fill_(0)
        g.replay()
        torch.cuda.synchronize()
        return (out.cpu().numpy().view(np.uint16), row.cpu().numpy(), ln.cpu().numpy())

    g1 = capture()
    _same_as_oracle(replay(g1), fg1_tok, fg1_len, F1_host, T_host, tok)
    scone.scone_table_rebuild_noalloc(table, fg2_tok, fg2_len, F2)
    g2 = capture()
    got = replay(g2)
    _same_as_oracle(got, fg2_tok, fg2_len, F2_host, T_host, tok)
    fresh = scone.scone_table_build(fg2_tok, fg2_len, BASE.K, BASE.vocab, BASE.d, F2, T)
    for x, y in zip(got, run_embed(fresh, tok, BASE.d)):
        assert np.array_equal(x, y)
    fresh.close()
    del g1, g2
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
    need = lambda n: 256 + -(-n // 256) * 256 + -(-(n * 4 * K) // 256) * 256
    n_under = (scratch - 768) // (4 * K + 1)            # SCONE_REBUILD_MAX_FGRAMS(3)
    n_over = n_under + 1
    while need(n_over) <= scratch:                      # the first size the header's rule refuses
        n_over += 1
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


def test_rebuild_noalloc_drops_the_suffix_index():
    """A built K = 3 table carries a suffix index (here with marker slots, as
    a third of the 2-grams are left out of the list); the rebuilt table has
    none, and every copy mode, the pipelined one included, still gives the
    oracle's answer on both."""
    fg1_tok, fg1_len, _ = synth.fgram_set(BASE)
    keep = ~((fg1_len == 2) & (np.arange(fg1_len.shape[0]) % 3 == 0))
    fg1_tok, fg1_len = fg1_tok[keep], fg1_len[keep]
    fg2_tok, fg2_len, _ = synth.fgram_set(OTHER)
    T_host = synth.rows_cpu(synth.T_seed(BASE), BASE.d, np.arange(BASE.vocab))
    F1_host = synth.rows_cpu(synth.F_seed(BASE), BASE.d, np.arange(fg1_len.shape[0]))
    F2_host = synth.rows_cpu(synth.F_seed(OTHER), OTHER.d, np.arange(OTHER.n_fgrams))
    T, F1, F2 = dev_rows(T_host), dev_rows(F1_host), dev_rows(F2_host)
    tok = synth.query_tokens(BASE)
    table = scone.scone_table_build(fg1_tok, fg1_len, BASE.K, BASE.vocab, BASE.d, F1, T)
    _, _, ml = scone.scone_fgram_suffix_index(fg1_tok, fg1_len, BASE.K)
    assert len(ml) > 0 and table.info()["n_markers"] == len(ml)
    modes = (scone.SCONE_COPY_AUTO, scone.SCONE_COPY_PIPELINED, scone.SCONE_COPY_REGISTERS)
    for mode in modes:
        scone.scone_table_set_copy_mode(table, mode)
        _same_as_oracle(run_embed(table, tok, BASE.d), fg1_tok, fg1_len, F1_host, T_host, tok)
    assert _rebuild_via_c_abi(table, fg2_tok, fg2_len, F2) == scone.SCONE_OK
    assert table.info()["n_markers"] == 0
    for mode in modes:
        scone.scone_table_set_copy_mode(table, mode)
        _same_as_oracle(run_embed(table, tok, BASE.d), fg2_tok, fg2_len, F2_host, T_host, tok)
    assert scone.scone_status(table) == scone.SCONE_OK
    table.close()
