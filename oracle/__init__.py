"""CPU oracles for SCONE's input embedding (Algorithm 1) and for the
construction of its f-gram set (Algorithm 3).

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import this package. The product path
(``paper_2502_01637_gb300``) never imports it and has no CPU fallback.

The arithmetic lives in ``scone_oracle.cpp`` (plain C++: a ``std::map`` keyed
by the exact token tuple, scanned as Algorithm 1 states) and
``discover_oracle.cpp`` (every n-gram counted in a ``std::map``, sorted as
Algorithm 3 states); this file only marshals numpy arrays through ctypes. ``__graft_entry__.build()`` compiles
``liboracle.so`` next to this file.
"""

from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
# SCONE_ORACLE_LIB points the pins at a deliberately broken copy (mutation tests).
_LIB_PATH = os.environ.get("SCONE_ORACLE_LIB") or os.path.join(_HERE, "liboracle.so")
_lib = None

OK = 0
ERR_INVALID_ARG = -1
ERR_TOKEN_RANGE = -2
ERR_DUPLICATE_FGRAM = -3

_i32p = ctypes.POINTER(ctypes.c_int32)
_i64p = ctypes.POINTER(ctypes.c_int64)
_u8p = ctypes.POINTER(ctypes.c_uint8)
_u16p = ctypes.POINTER(ctypes.c_uint16)
_u32p = ctypes.POINTER(ctypes.c_uint32)


def _load():
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError(f"oracle library missing: {_LIB_PATH} (run __graft_entry__.build())")
    lib = ctypes.CDLL(_LIB_PATH)
    lib.oracle_table_create.argtypes = [_i32p, _u8p, ctypes.c_int64, ctypes.c_int32,
                                        ctypes.c_int32, ctypes.POINTER(ctypes.c_void_p)]
    lib.oracle_table_create.restype = ctypes.c_int
    lib.oracle_table_destroy.argtypes = [ctypes.c_void_p]
    lib.oracle_table_destroy.restype = None
    lib.oracle_table_size.argtypes = [ctypes.c_void_p]
    lib.oracle_table_size.restype = ctypes.c_int64
    lib.oracle_select.argtypes = [ctypes.c_void_p, _i32p, ctypes.c_int32, ctypes.c_int32,
                                  _i64p, _u8p, _i64p]
    lib.oracle_select.restype = ctypes.c_int
    lib.oracle_select_at.argtypes = [ctypes.c_void_p, _i32p, ctypes.c_int32, ctypes.c_int32,
                                     _i64p, ctypes.c_int64, _i64p, _u8p]
    lib.oracle_select_at.restype = ctypes.c_int
    lib.oracle_embed.argtypes = [ctypes.c_void_p, _i32p, ctypes.c_int32, ctypes.c_int32,
                                 _u16p, ctypes.c_int64, _u16p, ctypes.c_int32, _u16p, _i64p, _u8p]
    lib.oracle_embed.restype = ctypes.c_int
    lib.oracle_embed_threads.argtypes = lib.oracle_embed.argtypes + [ctypes.c_int32]
    lib.oracle_embed_threads.restype = ctypes.c_int
    lib.oracle_decode.argtypes = [ctypes.c_void_p, ctypes.c_int32, _i32p, ctypes.c_int32, _i32p,
                                  ctypes.c_int32, _i32p, _u16p, ctypes.c_int64, _u16p,
                                  ctypes.c_int32, _u16p, _i64p, _u8p]
    lib.oracle_decode.restype = ctypes.c_int
    lib.oracle_discover.argtypes = [_i32p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                    ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, _i32p, _u8p,
                                    _u32p, ctypes.c_int64, _i64p, _i64p, _i64p]
    lib.oracle_discover.restype = ctypes.c_int
    lib.oracle_count_ngrams.argtypes = [_i32p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                        _i32p, _u8p, ctypes.c_int64, _i64p, _i64p,
                                        ctypes.c_int32]
    lib.oracle_count_ngrams.restype = ctypes.c_int
    _lib = lib
    return lib


def _ptr(a: np.ndarray, t):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(t)


class OracleError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: oracle status {code}")
        self.code = code


class Oracle:
    """V_fgram as an exact-tuple map, plus Algorithm 1 over token arrays.

    ``fgram_tok`` is ``[N, K]`` int32 (row-padded), ``fgram_len`` ``[N]`` with
    values in ``[2, K]``; row ``r`` of F belongs to f-gram ``r``.
    """

    def __init__(self, fgram_tok: np.ndarray, fgram_len: np.ndarray, K: int, vocab: int):
        lib = _load()
        self.K, self.vocab = int(K), int(vocab)
        self.fgram_tok = np.ascontiguousarray(fgram_tok, dtype=np.int32).reshape(-1, self.K)
        self.fgram_len = np.ascontiguousarray(fgram_len, dtype=np.uint8).reshape(-1)
        n = self.fgram_len.shape[0]
        h = ctypes.c_void_p()
        rc = lib.oracle_table_create(_ptr(self.fgram_tok, _i32p), _ptr(self.fgram_len, _u8p),
                                     n, self.K, self.vocab, ctypes.byref(h))
        if rc != OK:
            raise OracleError(rc, "oracle_table_create")
        self._h = h
        self.n_fgrams = n

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and h.value and _lib is not None:
            _lib.oracle_table_destroy(h)
            self._h = None

    def size(self) -> int:
        return int(_load().oracle_table_size(self._h))

    def select(self, tok: np.ndarray):
        """Returns (row int64 [B,L], len uint8 [B,L], queries int64 [B,L], status)."""
        tok = np.ascontiguousarray(tok, dtype=np.int32)
        B, L = tok.shape
        row = np.empty((B, L), np.int64)
        ln = np.empty((B, L), np.uint8)
        q = np.empty((B, L), np.int64)
        rc = _load().oracle_select(self._h, _ptr(tok, _i32p), B, L, _ptr(row, _i64p),
                                   _ptr(ln, _u8p), _ptr(q, _i64p))
        if rc not in (OK, ERR_TOKEN_RANGE):
            raise OracleError(rc, "oracle_select")
        return row, ln, q, rc

    def select_at(self, tok: np.ndarray, positions: np.ndarray):
        """Selection at flattened positions only. Returns (row, len, status)."""
        tok = np.ascontiguousarray(tok, dtype=np.int32)
        B, L = tok.shape
        pos = np.ascontiguousarray(positions, dtype=np.int64)
        row = np.empty(pos.shape[0], np.int64)
        ln = np.empty(pos.shape[0], np.uint8)
        rc = _load().oracle_select_at(self._h, _ptr(tok, _i32p), B, L, _ptr(pos, _i64p),
                                      pos.shape[0], _ptr(row, _i64p), _ptr(ln, _u8p))
        if rc not in (OK, ERR_TOKEN_RANGE):
            raise OracleError(rc, "oracle_select_at")
        return row, ln, rc

    def embed(self, tok: np.ndarray, F: np.ndarray, T: np.ndarray, threads: int = 1):
        """Algorithm 1 output. F [N,d], T [vocab,d] as uint16 (raw bf16 words).
        threads > 1 splits the sequences over that many std::threads.

        Returns (out uint16 [B,L,d], row int64 [B,L], len uint8 [B,L], status).
        """
        tok = np.ascontiguousarray(tok, dtype=np.int32)
        B, L = tok.shape
        F = np.ascontiguousarray(F, dtype=np.uint16)
        T = np.ascontiguousarray(T, dtype=np.uint16)
        d = T.shape[1]
        assert F.ndim == 2 and (F.shape[0] == 0 or F.shape[1] == d)
        out = np.empty((B, L, d), np.uint16)
        row = np.empty((B, L), np.int64)
        ln = np.empty((B, L), np.uint8)
        Fp = F if F.size else np.zeros((1, d), np.uint16)
        args = (self._h, _ptr(tok, _i32p), B, L, _ptr(Fp, _u16p), F.shape[0], _ptr(T, _u16p), d,
                _ptr(out, _u16p), _ptr(row, _i64p), _ptr(ln, _u8p))
        rc = (_load().oracle_embed_threads(*args, int(threads)) if threads > 1
              else _load().oracle_embed(*args))
        if rc not in (OK, ERR_TOKEN_RANGE):
            raise OracleError(rc, "oracle_embed")
        return out, row, ln, rc

    def decode(self, hist: np.ndarray, hist_len: np.ndarray, new_tok: np.ndarray,
               F: np.ndarray, T: np.ndarray):
        """Decode steps. hist [S,H] (right-aligned prefixes), hist_len [S],
        new_tok [steps,S]. Returns (out [steps,S,d], row [steps,S], len, status).
        """
        hist = np.ascontiguousarray(hist, dtype=np.int32)
        S, H = hist.shape
        hl = np.ascontiguousarray(hist_len, dtype=np.int32)
        nt = np.ascontiguousarray(new_tok, dtype=np.int32)
        steps = nt.shape[0]
        F = np.ascontiguousarray(F, dtype=np.uint16)
        T = np.ascontiguousarray(T, dtype=np.uint16)
        d = T.shape[1]
        out = np.empty((steps, S, d), np.uint16)
        row = np.empty((steps, S), np.int64)
        ln = np.empty((steps, S), np.uint8)
        Fp = F if F.size else np.zeros((1, d), np.uint16)
        rc = _load().oracle_decode(self._h, S, _ptr(hist, _i32p), H, _ptr(hl, _i32p), steps,
                                   _ptr(nt, _i32p), _ptr(Fp, _u16p), F.shape[0], _ptr(T, _u16p),
                                   d, _ptr(out, _u16p), _ptr(row, _i64p), _ptr(ln, _u8p))
        if rc not in (OK, ERR_TOKEN_RANGE):
            raise OracleError(rc, "oracle_decode")
        return out, row, ln, rc


def discover(tok: np.ndarray, K: int, vocab: int, S: int, min_count: int = 1):
    """Algorithm 3 on a [B, L] corpus: the S most frequent n-grams, n = 2..K,
    among those appearing at least ``min_count`` times; ties by length, then
    first occurrence. Listed by length, then first occurrence.

    Returns a dict: ``tok`` [n, K] int32 padded with -1, ``len`` [n] uint8,
    ``count`` [n] uint32, ``distinct`` and ``frequent`` ([K + 1] int64: per
    length, the n-grams that appear and those reaching ``min_count``).
    """
    tok = np.ascontiguousarray(tok, dtype=np.int32)
    B, L = tok.shape
    cap = int(min(S, B * max(L - 1, 0) * (K - 1)))
    out_tok = np.empty((max(cap, 1), K), np.int32)
    out_len = np.empty(max(cap, 1), np.uint8)
    out_cnt = np.empty(max(cap, 1), np.uint32)
    n_out = ctypes.c_int64()
    distinct = np.zeros(K + 1, np.int64)
    frequent = np.zeros(K + 1, np.int64)
    tp = _ptr(tok, _i32p) if tok.size else None
    rc = _load().oracle_discover(tp, B, L, vocab, K, S, min_count, _ptr(out_tok, _i32p),
                                 _ptr(out_len, _u8p), _ptr(out_cnt, _u32p), cap,
                                 ctypes.byref(n_out), _ptr(distinct, _i64p),
                                 _ptr(frequent, _i64p))
    if rc != OK:
        raise OracleError(rc, "oracle_discover")
    n = n_out.value
    return {"tok": out_tok[:n].copy(), "len": out_len[:n].copy(), "count": out_cnt[:n].copy(),
            "distinct": distinct, "frequent": frequent}


def count_ngrams(tok: np.ndarray, K: int, q_tok: np.ndarray, q_len: np.ndarray, threads: int = 0):
    """Occurrences of each (distinct) query n-gram in a [B, L] corpus: every
    window is looked up in a map of the queries. Returns (count int64 [nq],
    first occurrence int64 [nq]); threads = 0 uses every core."""
    tok = np.ascontiguousarray(tok, dtype=np.int32)
    B, L = tok.shape
    q_tok = np.ascontiguousarray(q_tok, dtype=np.int32).reshape(-1, K)
    q_len = np.ascontiguousarray(q_len, dtype=np.uint8).reshape(-1)
    nq = q_len.shape[0]
    counts = np.empty(max(nq, 1), np.int64)
    first = np.empty(max(nq, 1), np.int64)
    rc = _load().oracle_count_ngrams(_ptr(tok, _i32p), B, L, K, _ptr(q_tok, _i32p),
                                     _ptr(q_len, _u8p), nq, _ptr(counts, _i64p),
                                     _ptr(first, _i64p), threads)
    if rc != OK:
        raise OracleError(rc, "oracle_count_ngrams")
    return counts[:nq], first[:nq]
