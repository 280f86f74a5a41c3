"""The suffix index a table build adds (host code, no GPU): extension bits and
marker n-grams against a brute-force reading of their definition, and the
argument and duplicate checks."""
import numpy as np
import pytest

import paper_2502_01637_gb300 as scone

pytestmark = pytest.mark.filterwarnings("ignore")


def brute_force(ft, fl):
    """ext[r]: f-gram r is the suffix of a longer listed f-gram. Markers: the
    suffixes (length >= 2) of listed f-grams that are not listed, in the order
    f-gram 0, 1, ... reaches them, longest suffix first."""
    grams = [tuple(int(x) for x in ft[r, :fl[r]]) for r in range(len(fl))]
    listed = {g: r for r, g in enumerate(grams)}
    ext = np.zeros(len(grams), np.uint8)
    for g in grams:
        for m in range(2, len(g)):
            s = g[len(g) - m:]
            if s in listed:
                ext[listed[s]] = 1
    markers, seen = [], set()
    for g in grams:
        for m in range(len(g) - 1, 1, -1):
            s = g[len(g) - m:]
            if s not in listed and s not in seen:
                seen.add(s)
                markers.append(s)
    return ext, markers


def random_list(rng, n, K, vocab):
    """Distinct n-grams of lengths 2..K over a small vocabulary, so that many
    suffixes coincide with listed f-grams and with one another."""
    out, seen = [], set()
    while len(out) < n:
        ln = int(rng.integers(2, K + 1))
        g = tuple(int(x) for x in rng.integers(0, vocab, ln))
        if g not in seen:
            seen.add(g)
            out.append(g)
    ft = np.full((n, K), -1, np.int32)
    fl = np.zeros(n, np.uint8)
    for r, g in enumerate(out):
        ft[r, :len(g)] = g
        fl[r] = len(g)
    return ft, fl


@pytest.mark.parametrize("K,vocab,n,seed", [(3, 6, 150, 1), (5, 5, 800, 2), (5, 40, 3000, 3),
                                            (8, 4, 2000, 4), (4, 1000, 500, 5)])
def test_matches_brute_force(K, vocab, n, seed):
    ft, fl = random_list(np.random.default_rng(seed), n, K, vocab)
    ext, mt, ml = scone.scone_fgram_suffix_index(ft, fl, K)
    o_ext, o_markers = brute_force(ft, fl)
    assert np.array_equal(ext, o_ext)
    got = [tuple(int(x) for x in mt[i, :ml[i]]) for i in range(len(ml))]
    assert got == o_markers
    assert (mt[np.arange(mt.shape[1])[None, :] >= ml[:, None]] == -1).all()   # padding


def test_closure_property():
    """After adding the markers every suffix of every entry is present."""
    ft, fl = random_list(np.random.default_rng(7), 2000, 5, 30)
    ext, mt, ml = scone.scone_fgram_suffix_index(ft, fl, 5)
    entries = {tuple(ft[r, :fl[r]]) for r in range(len(fl))}
    entries |= {tuple(mt[i, :ml[i]]) for i in range(len(ml))}
    for g in entries:
        for m in range(2, len(g)):
            assert g[len(g) - m:] in entries


def test_worked_example():
    """(1 2 3 4) needs its suffixes (2 3 4) and (3 4): (3 4) is listed and
    gets the bit, (2 3 4) becomes a marker; (5 3 4) reaches (3 4) again."""
    ft = np.array([[1, 2, 3, 4], [3, 4, -1, -1], [5, 3, 4, -1], [7, 8, -1, -1]], np.int32)
    fl = np.array([4, 2, 3, 2], np.uint8)
    ext, mt, ml = scone.scone_fgram_suffix_index(ft, fl, 4)
    assert ext.tolist() == [0, 1, 0, 0]
    assert ml.tolist() == [3] and mt.tolist() == [[2, 3, 4, -1]]


def test_k2_and_empty_lists_have_no_markers():
    ft = np.array([[1, 2], [2, 3]], np.int32)
    ext, mt, ml = scone.scone_fgram_suffix_index(ft, np.array([2, 2], np.uint8), 2)
    assert ext.tolist() == [0, 0] and len(ml) == 0
    ext, mt, ml = scone.scone_fgram_suffix_index(np.zeros((0, 3), np.int32),
                                                 np.zeros(0, np.uint8), 3)
    assert len(ext) == 0 and len(ml) == 0


def test_count_only_and_partial_capacity():
    import ctypes
    lib = scone.load_library()
    ft, fl = random_list(np.random.default_rng(9), 400, 5, 8)
    _, o_markers = brute_force(ft, fl)
    assert len(o_markers) > 3
    cnt = ctypes.c_int64(-1)
    mt = np.full((2, 5), 77, np.int32)
    ml = np.zeros(2, np.uint8)
    rc = lib.scone_fgram_suffix_index(ft.ctypes.data, fl.ctypes.data, len(fl), 5, None,
                                      mt.ctypes.data, ml.ctypes.data, 2, ctypes.byref(cnt))
    assert rc == 0 and cnt.value == len(o_markers)
    for i in range(2):
        assert tuple(mt[i, :ml[i]]) == o_markers[i]


def test_errors():
    import ctypes
    lib = scone.load_library()
    cnt = ctypes.c_int64(0)
    ft = np.array([[1, 2, 3], [1, 2, 3]], np.int32)
    fl = np.array([3, 3], np.uint8)
    with pytest.raises(scone.SconeError) as e:
        scone.scone_fgram_suffix_index(ft, fl, 3)
    assert e.value.code == scone.SCONE_ERR_DUPLICATE_FGRAM
    inv = scone.SCONE_ERR_INVALID_ARG
    bad_len = np.array([3, 4], np.uint8)
    assert lib.scone_fgram_suffix_index(ft.ctypes.data, bad_len.ctypes.data, 2, 3, None, None,
                                        None, 0, ctypes.byref(cnt)) == inv
    assert lib.scone_fgram_suffix_index(ft.ctypes.data, fl.ctypes.data, 2, 9, None, None, None,
                                        0, ctypes.byref(cnt)) == inv
    assert lib.scone_fgram_suffix_index(ft.ctypes.data, fl.ctypes.data, 2, 3, None, None, None,
                                        0, None) == inv
    assert lib.scone_fgram_suffix_index(None, None, 2, 3, None, None, None, 0,
                                        ctypes.byref(cnt)) == inv
    assert lib.scone_fgram_suffix_index(ft.ctypes.data, fl.ctypes.data, 2, 3, None, None, None,
                                        4, ctypes.byref(cnt)) == inv
