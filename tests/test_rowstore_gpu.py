"""The row store (F in a file, rows cached in HBM) against the oracle (GPU).

F is written to a file in the test's temporary directory; the table's F
pointer is a small dummy, so every F row the output holds came through the
store (cache hit or file read). A cache much smaller than F forces misses,
evictions and slot conflicts; repeating a batch turns misses into hits.
Outputs must equal the oracle's bytes exactly.
"""

import os

import numpy as np
import pytest
import torch

import synth
import paper_2502_01637_gb300 as scone
from gpu_cases import DEV, SmallCase, dev_rows

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS["tiny"].scaled("rowstore", B=6, L=700, d=64, quotas=((2, 6000), (3, 4000)))


@pytest.fixture(scope="module")
def case(tmp_path_factory):
    c = SmallCase(W)
    path = os.path.join(str(tmp_path_factory.mktemp("rows")), "F.bin")
    c.F.tofile(path)
    # the table's own F is never read by the store path: a one-row stand-in
    c.table = scone.scone_table_build(c.fg_tok, c.fg_len, W.K, W.vocab, W.d,
                                      dev_rows(c.F[:1]), dev_rows(c.T))
    c.path = path
    yield c
    c.table.close()


def gather(case, store, tok):
    t = torch.from_numpy(np.ascontiguousarray(tok, np.int32)).to(DEV)
    n = t.numel()
    row = torch.empty(n, dtype=torch.int32, device=DEV)
    out = torch.empty((n, W.d), dtype=torch.int16, device=DEV)
    scone.scone_match(case.table, t, row)
    scone.scone_rowstore_gather(store, case.table, t.reshape(-1), row, out)
    scone.scone_status(case.table)
    return out.cpu().numpy().view(np.uint16)


def test_matches_oracle_with_small_cache(case):
    store = scone.RowStore(case.path, case.F.shape[0], W.d, cache_rows=97, threads=4)
    exp, _, _, rc = case.expected()
    assert rc == 0
    exp = exp.reshape(-1, W.d)
    got = gather(case, store, case.tok)
    assert np.array_equal(got, exp)
    s1 = store.stats()
    assert s1["misses"] > 0 and s1["rows_read"] > 0
    got2 = gather(case, store, case.tok)            # same batch again: hot rows now cached
    assert np.array_equal(got2, exp)
    s2 = store.stats()
    assert s2["misses"] - s1["misses"] < s1["misses"]
    store.close()


def test_large_cache_reads_each_row_once(case):
    store = scone.RowStore(case.path, case.F.shape[0], W.d, cache_rows=1 << 16, threads=2)
    exp = case.expected()[0].reshape(-1, W.d)
    for _ in range(3):
        assert np.array_equal(gather(case, store, case.tok), exp)
    s = store.stats()
    # a cache much larger than the rows used: each distinct row read once,
    # unless two of them share a slot
    used = np.unique(case.expected()[1][case.expected()[1] >= 0])
    assert s["rows_read"] <= used.size * 1.05 and s["rows_read"] >= used.size * 0.9
    store.close()


def test_decode_selection_then_store(case):
    """scone_decode_step without rows (out = NULL) then the store equals the
    fused decode step over the table's full F."""
    full = scone.scone_table_build(case.fg_tok, case.fg_len, W.K, W.vocab, W.d, dev_rows(case.F),
                                   dev_rows(case.T))
    store = scone.RowStore(case.path, case.F.shape[0], W.d, cache_rows=211)
    S, H = 64, W.K - 1
    hist = case.tok[:, :H].repeat(11, axis=0)[:S]
    hl = np.full(S, H, np.int32)
    a = scone.scone_decode_create(full, hist, hl)
    b = scone.scone_decode_create(case.table, hist, hl)
    for k in range(5):
        new = torch.from_numpy(np.ascontiguousarray(case.tok.reshape(-1)[k * S:(k + 1) * S]))
        new = new.to(DEV)
        out_a = torch.empty((S, W.d), dtype=torch.int16, device=DEV)
        scone.scone_decode_step(a, new, out_a)
        row_b = torch.empty(S, dtype=torch.int32, device=DEV)
        lib = scone.load_library()
        assert lib.scone_decode_step(b.handle, new.data_ptr(), None, row_b.data_ptr(), None,
                                     torch.cuda.current_stream().cuda_stream) == 0
        out_b = torch.empty((S, W.d), dtype=torch.int16, device=DEV)
        scone.scone_rowstore_gather(store, case.table, new, row_b, out_b)
        assert torch.equal(out_a, out_b), k
    a.close()
    b.close()
    store.close()
    full.close()


def test_errors(case, tmp_path):
    with pytest.raises(scone.SconeError):
        scone.RowStore(case.path, case.F.shape[0] + 1, W.d, 16)      # file too short
    with pytest.raises(scone.SconeError):
        scone.RowStore(str(tmp_path / "missing.bin"), 10, W.d, 16)
    store = scone.RowStore(case.path, 100, W.d, 16)                 # rows >= 100 are invalid
    t = torch.from_numpy(case.tok[0]).to(DEV)
    row = torch.empty(t.numel(), dtype=torch.int32, device=DEV)
    scone.scone_match(case.table, t, row)
    assert int((row >= 100).sum()) > 0
    out = torch.empty((t.numel(), W.d), dtype=torch.int16, device=DEV)
    scone.scone_rowstore_gather(store, case.table, t, row, out)
    assert scone.scone_status(case.table, raise_on_error=False) == scone.SCONE_ERR_INVALID_ARG
    store.close()


def test_direct_io_rows(tmp_path):
    """4 KiB rows (d = 2048): the store reads the file with O_DIRECT where the
    filesystem allows it; bytes still equal the oracle's."""
    w = synth.WORKLOADS["tiny"].scaled("rowstore_4k", B=2, L=300, d=2048,
                                       quotas=((2, 1500), (3, 1000)))
    c = SmallCase(w)
    path = str(tmp_path / "F4k.bin")
    c.F.tofile(path)
    table = scone.scone_table_build(c.fg_tok, c.fg_len, w.K, w.vocab, w.d, dev_rows(c.F[:1]),
                                    dev_rows(c.T))
    store = scone.RowStore(path, c.F.shape[0], w.d, cache_rows=50, threads=3)
    t = torch.from_numpy(c.tok).to(DEV)
    row = torch.empty(t.numel(), dtype=torch.int32, device=DEV)
    out = torch.empty((t.numel(), w.d), dtype=torch.int16, device=DEV)
    scone.scone_match(table, t, row)
    scone.scone_rowstore_gather(store, table, t.reshape(-1), row, out)
    scone.scone_status(table)
    exp = c.expected()[0].reshape(-1, w.d)
    assert np.array_equal(out.cpu().numpy().view(np.uint16), exp)
    assert store.stats()["rows_read"] > 0
    store.close()
    table.close()


def test_long_keys_and_k8(tmp_path):
    """A table with 32-byte slots (K = 8 over a 2^20-token vocabulary): rows
    selected by the long-key matcher and served by the store equal the
    oracle's bytes."""
    w = synth.Workload("rowstore_k8", 88, 1 << 20, 1.05, 3, 600,
                       tuple((n, 1200) for n in range(2, 9)), 8, 64, inject_p=0.05,
                       n_phrases=256, phrase_len=(8, 10))
    c = SmallCase(w)
    path = str(tmp_path / "F8.bin")
    c.F.tofile(path)
    table = scone.scone_table_build(c.fg_tok, c.fg_len, w.K, w.vocab, w.d, dev_rows(c.F[:1]),
                                    dev_rows(c.T))
    assert table.info()["slot_bytes"] == 32
    store = scone.RowStore(path, c.F.shape[0], w.d, cache_rows=61, threads=2)
    t = torch.from_numpy(c.tok).to(DEV)
    row = torch.empty(t.numel(), dtype=torch.int32, device=DEV)
    out = torch.empty((t.numel(), w.d), dtype=torch.int16, device=DEV)
    scone.scone_match(table, t, row)
    scone.scone_rowstore_gather(store, table, t.reshape(-1), row, out)
    scone.scone_status(table)
    exp_out, exp_row, exp_len, _ = c.expected()
    assert np.array_equal(row.cpu().numpy(), exp_row.reshape(-1).astype(np.int32))
    assert np.array_equal(out.cpu().numpy().view(np.uint16), exp_out.reshape(-1, w.d))
    assert (exp_len == 8).any()
    store.close()
    table.close()


def test_probe_reads_reports_the_file_rate(case):
    """The storage probe reads rows of the store's own file (no GPU work, no
    cache change) and reports positive rates that agree with each other."""
    store = scone.RowStore(case.path, W.n_fgrams, W.d, 64, threads=4)
    before = store.stats()
    r = scone.scone_rowstore_probe_reads(store, 2000, seed=3)
    assert r["rows_per_s"] > 0
    assert abs(r["bytes_per_s"] / r["rows_per_s"] - W.d * 2) < 1e-6 * W.d * 2
    assert store.stats() == before                 # the gather statistics are untouched
    out = gather(case, store, case.tok)            # the store still gathers exactly
    o_out, _, _, _ = case.expected()
    assert np.array_equal(out, o_out.reshape(out.shape))
    with pytest.raises(scone.SconeError):
        scone.scone_rowstore_probe_reads(store, 0)
    store.close()
