"""Seeded synthetic inputs for the SCONE embedding path.

Shared by both sides of every parity check: it produces token streams, f-gram
lists and bf16 embedding rows, and holds none of the method's arithmetic (no
suffix matching, no lookup, no gather). ``synth.cpp`` / ``synth_rows.cu`` hold
the generators; this file defines the named workloads and marshals arrays.

Workloads (shapes of the paper's settings; the paper's corpora and trained
F are not available, so seeded Zipf streams stand in for them):

=================  =====  ====  ======  ===========  ===  ====  ==============
name               vocab  s     B x L   f-grams      K    d     F location
=================  =====  ====  ======  ===========  ===  ====  ==============
tiny               32000  1.1   4x512   1e5 (60/40)  3    256   device
prefill_1b         1e5    1.1   32x2048 1e6 (60/40)  3    2048  device
large_hbm          1e5    1.1   64x4096 1e7 (60/40)  3    2048  device
offload_decode     1e5    1.1   512 seq x 256 steps  2e7  3     2048  host-mapped
stress_k5          1e5    1.05  16x8192 5e6 n=2..5   5    1536  device
prescan            1e5    1.1   2^19x2048 1e7 (60/40) 3   8     (tokens in host memory)
discover           1e5    1.1   2^19x2048 S = 1e7    3   -     (corpus in HBM)
discover_k5        1e5    1.05  2^17x2048 S = 5e6    5   -     (corpus in HBM)
=================  =====  ====  ======  ===========  ===  ====  ==============

f-gram sets are the first distinct n-grams of a separate Zipf source stream of
the same law (per-length quotas), row id = first-seen order. The stress
workload injects repeated phrases (pool of 4096 phrases, lengths U[4,8],
Zipf(1.05) tokens) at a start rate of 0.05/6 per position into both the
query and the source streams, so that 4- and 5-grams recur.
"""

from __future__ import annotations

import ctypes
import dataclasses
import functools
import os
from typing import Dict, Optional, Tuple

import numpy as np

MASTER_SEED = 20250203

# stream ids
S_QUERY, S_SOURCE, S_FROWS, S_TROWS, S_PHRASES, S_DEC_HIST, S_DEC_TOK, S_MODEL = range(8)

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libsynth.so")
_lib = None

_i32p = ctypes.POINTER(ctypes.c_int32)
_i64p = ctypes.POINTER(ctypes.c_int64)
_u8p = ctypes.POINTER(ctypes.c_uint8)
_u16p = ctypes.POINTER(ctypes.c_uint16)


def _load():
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError(f"synth library missing: {_LIB_PATH} (run __graft_entry__.build())")
    lib = ctypes.CDLL(_LIB_PATH)
    u64, i32, i64, dbl = ctypes.c_uint64, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
    lib.synth_mix64.argtypes = [u64]
    lib.synth_mix64.restype = u64
    lib.synth_draw.argtypes = [u64, u64]
    lib.synth_draw.restype = u64
    lib.synth_stream_seed.argtypes = [u64, ctypes.c_uint32, ctypes.c_uint32, u64]
    lib.synth_stream_seed.restype = u64
    lib.synth_zipf_tokens.argtypes = [u64, i32, dbl, i64, dbl, _i32p, _i32p, i32, i32, _i32p]
    lib.synth_zipf_tokens.restype = ctypes.c_int
    lib.synth_query_batch.argtypes = [u64, ctypes.c_uint32, ctypes.c_uint32, u64, i64, i64, i32,
                                      dbl, dbl, _i32p, _i32p, i32, i32, _i32p, i32]
    lib.synth_query_batch.restype = ctypes.c_int
    lib.synth_phrase_pool.argtypes = [u64, i32, dbl, i32, i32, i32, _i32p, _i32p]
    lib.synth_phrase_pool.restype = ctypes.c_int
    lib.synth_fgram_set.argtypes = [u64, i32, dbl, i32, _i64p, dbl, _i32p, _i32p, i32, i32, i64,
                                    _i32p, _u8p, _i64p, _i64p]
    lib.synth_fgram_set.restype = i64
    lib.synth_rows_cpu.argtypes = [u64, i32, _i64p, i64, _u16p]
    lib.synth_rows_cpu.restype = None
    lib.synth_rows_range_cpu.argtypes = [u64, i32, i64, i64, _u16p, i32]
    lib.synth_rows_range_cpu.restype = None
    lib.synth_rows_gpu.argtypes = [u64, i32, i64, i64, ctypes.c_void_p, ctypes.c_void_p]
    lib.synth_rows_gpu.restype = ctypes.c_int
    _lib = lib
    return lib


def _p(a, t):
    return None if a is None else a.ctypes.data_as(t)


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    wid: int                 # workload id, mixed into every seed
    vocab: int
    zipf_s: float
    B: int                   # sequences (prefill) ...
    L: int                   # ... of L tokens
    quotas: Tuple[Tuple[int, int], ...]   # ((n, count), ...)
    K: int
    d: int
    location: str = "device"             # "device" or "host_mapped"
    inject_p: float = 0.0                # phrase start probability per position
    n_phrases: int = 0
    phrase_len: Tuple[int, int] = (4, 8)
    load_factor: float = 0.5
    dec_S: int = 0                       # decode: live sequences
    dec_hist: int = 0                    # decode: history tokens per sequence
    dec_steps: int = 0                   # decode: steps
    min_count: int = 5                   # f-gram discovery: eligibility threshold (Sec. 3.2)
    # order of the f-gram list (row r of F belongs to f-gram r): "first_seen" in
    # the source stream, or "count": by descending count in the source stream
    # (ties in first-seen order), the order a top-S-by-count selection yields
    row_order: str = "first_seen"

    @property
    def n_fgrams(self) -> int:
        return sum(c for _, c in self.quotas)

    @property
    def n_tokens(self) -> int:
        return self.B * self.L

    def scaled(self, name: str, **kw) -> "Workload":
        """A smaller variant with the same laws (for tests)."""
        return dataclasses.replace(self, name=name, **kw)


def _split(n: int, parts: Dict[int, float]) -> Tuple[Tuple[int, int], ...]:
    out, acc = [], 0
    items = sorted(parts.items())
    for k, (length, frac) in enumerate(items):
        c = n - acc if k == len(items) - 1 else int(round(n * frac))
        out.append((length, c))
        acc += c
    return tuple(out)


WORKLOADS: Dict[str, Workload] = {
    "tiny": Workload("tiny", 1, 32000, 1.1, 4, 512, ((2, 60000), (3, 40000)), 3, 256),
    "prefill_1b": Workload("prefill_1b", 2, 100000, 1.1, 32, 2048,
                           _split(1_000_000, {2: 0.6, 3: 0.4}), 3, 2048),
    "large_hbm": Workload("large_hbm", 3, 100000, 1.1, 64, 4096,
                          _split(10_000_000, {2: 0.6, 3: 0.4}), 3, 2048),
    "offload_decode": Workload("offload_decode", 4, 100000, 1.1, 0, 0,
                               _split(20_000_000, {2: 0.6, 3: 0.4}), 3, 2048,
                               location="host_mapped", dec_S=512, dec_hist=2, dec_steps=256,
                               row_order="count"),
    "stress_k5": Workload("stress_k5", 5, 100000, 1.05, 16, 8192,
                          ((2, 1_666_666), (3, 1_666_666), (4, 833_334), (5, 833_334)), 5, 1536,
                          inject_p=0.05 / 6, n_phrases=4096),
    # training-time pre-scan (tag every corpus token with its match length and row):
    # 2^19 training sequences of 2048 tokens (1.07e9 tokens) in host memory
    "prescan": Workload("prescan", 6, 100000, 1.1, 1 << 19, 2048,
                        _split(10_000_000, {2: 0.6, 3: 0.4}), 3, 8, location="host_mapped"),
    # f-gram discovery (Algorithm 3 by K-1 scans): the 1e7 most frequent 2..3-grams
    # (count >= 5) of a 1.07e9-token corpus (2^19 sequences of 2048) held in HBM;
    # the quotas give S and its split is not used
    "discover": Workload("discover", 7, 100000, 1.1, 1 << 19, 2048,
                         _split(10_000_000, {2: 0.6, 3: 0.4}), 3, 8),
    # the same with K = 5 over the stress law (phrases injected, so 4- and 5-grams recur)
    "discover_k5": Workload("discover_k5", 8, 100000, 1.05, 1 << 17, 2048,
                            _split(5_000_000, {2: 0.5, 3: 0.5}), 5, 8,
                            inject_p=0.05 / 6, n_phrases=4096),
}


def stream_seed(w: Workload, stream_id: int, sub: int = 0) -> int:
    return int(_load().synth_stream_seed(MASTER_SEED, w.wid, stream_id, sub))


def F_seed(w: Workload) -> int:
    return stream_seed(w, S_FROWS)


def T_seed(w: Workload) -> int:
    return stream_seed(w, S_TROWS)


@functools.lru_cache(maxsize=8)
def phrase_pool(w: Workload):
    """(tok [n_phrases, max_len] int32 padded with -1, len [n_phrases] int32)."""
    if w.n_phrases == 0:
        return None, None
    lo, hi = w.phrase_len
    tok = np.empty((w.n_phrases, hi), np.int32)
    ln = np.empty(w.n_phrases, np.int32)
    rc = _load().synth_phrase_pool(stream_seed(w, S_PHRASES), w.vocab, w.zipf_s, w.n_phrases,
                                   lo, hi, _p(tok, _i32p), _p(ln, _i32p))
    assert rc == 0
    return tok, ln


def zipf_tokens(w: Workload, seed: int, n: int, inject: bool = True) -> np.ndarray:
    out = np.empty(n, np.int32)
    pt, pl = phrase_pool(w) if inject else (None, None)
    n_ph = 0 if pt is None else pt.shape[0]
    stride = 0 if pt is None else pt.shape[1]
    rc = _load().synth_zipf_tokens(seed, w.vocab, w.zipf_s, n, w.inject_p if n_ph else 0.0,
                                   _p(pt, _i32p), _p(pl, _i32p), n_ph, stride, _p(out, _i32p))
    assert rc == 0
    return out


def query_tokens(w: Workload, seqs: Optional[range] = None, out: Optional[np.ndarray] = None,
                 threads: int = 0) -> np.ndarray:
    """Query batch [B, L] int32; sequence b is sub-stream b of the query stream.

    ``seqs`` must be a contiguous range; ``out`` may be a preallocated [len, L]
    int32 array (for instance a view of host-mapped memory).
    """
    seqs = range(w.B) if seqs is None else seqs
    assert seqs.step == 1
    if out is None:
        out = np.empty((len(seqs), w.L), np.int32)
    assert out.shape == (len(seqs), w.L) and out.dtype == np.int32 and out.flags["C_CONTIGUOUS"]
    pt, pl = phrase_pool(w)
    n_ph = 0 if pt is None else pt.shape[0]
    stride = 0 if pt is None else pt.shape[1]
    threads = threads or min(16, os.cpu_count() or 1)
    rc = _load().synth_query_batch(MASTER_SEED, w.wid, S_QUERY, seqs.start, len(seqs), w.L,
                                   w.vocab, w.zipf_s, w.inject_p if n_ph else 0.0, _p(pt, _i32p),
                                   _p(pl, _i32p), n_ph, stride, _p(out, _i32p), threads)
    assert rc == 0
    return out


_FGRAM_CACHE: Dict[Workload, tuple] = {}


def _fgram_set_first_seen(w: Workload, max_stream: int, with_counts: bool):
    quota = np.zeros(w.K + 1, np.int64)
    for n, c in w.quotas:
        quota[n] = c
    N = int(quota.sum())
    tok = np.empty((N, w.K), np.int32)
    ln = np.empty(N, np.uint8)
    counts = np.empty(N, np.int64) if with_counts else None
    used = ctypes.c_int64(0)
    pt, pl = phrase_pool(w)
    n_ph = 0 if pt is None else pt.shape[0]
    stride = 0 if pt is None else pt.shape[1]
    got = _load().synth_fgram_set(stream_seed(w, S_SOURCE), w.vocab, w.zipf_s, w.K,
                                  _p(quota, _i64p), w.inject_p if n_ph else 0.0, _p(pt, _i32p),
                                  _p(pl, _i32p), n_ph, stride, max_stream, _p(tok, _i32p),
                                  _p(ln, _u8p), ctypes.byref(used), _p(counts, _i64p))
    if got != N:
        raise RuntimeError(f"f-gram generation for {w.name} failed ({got})")
    return tok, ln, int(used.value), counts


def fgram_set(w: Workload, max_stream: int = 4_000_000_000):
    """(fgram_tok [N, K] int32 padded with -1, fgram_len [N] uint8, stream tokens used),
    listed in the workload's row order."""
    return _fgram_entry(w, max_stream)[:3]


def fgram_counts(w: Workload, max_stream: int = 4_000_000_000) -> np.ndarray:
    """Count of each f-gram of fgram_set(w) (same order) in the source stream."""
    e = _fgram_entry(w, max_stream, with_counts=True)
    return e[3]


def _fgram_entry(w: Workload, max_stream: int, with_counts: bool = False):
    e = _FGRAM_CACHE.get(w)
    if e is not None and (e[3] is not None or not with_counts):
        return e
    need_counts = with_counts or w.row_order == "count"
    tok, ln, used, counts = _fgram_set_first_seen(w, max_stream, need_counts)
    if w.row_order == "count":
        order = np.argsort(-counts, kind="stable")
        tok, ln, counts = tok[order], ln[order], counts[order]
    elif w.row_order != "first_seen":
        raise ValueError(f"unknown row order {w.row_order}")
    e = (tok, ln, used, counts)
    if len(_FGRAM_CACHE) >= 4:
        _FGRAM_CACHE.pop(next(iter(_FGRAM_CACHE)))
    _FGRAM_CACHE[w] = e
    return e


def rows_cpu(seed: int, d: int, row_ids) -> np.ndarray:
    """bf16 rows (raw uint16) for the given row ids, [len(row_ids), d]."""
    ids = np.ascontiguousarray(row_ids, dtype=np.int64).reshape(-1)
    out = np.empty((ids.shape[0], d), np.uint16)
    _load().synth_rows_cpu(seed, d, _p(ids, _i64p), ids.shape[0], _p(out, _u16p))
    return out


def rows_range_cpu(seed: int, d: int, row0: int, n: int, threads: int = 0) -> np.ndarray:
    out = np.empty((n, d), np.uint16)
    threads = threads or min(16, os.cpu_count() or 1)
    _load().synth_rows_range_cpu(seed, d, row0, n, _p(out, _u16p), threads)
    return out


def rows_gpu(seed: int, d: int, row0: int, n: int, out_ptr: int, stream_ptr: int) -> None:
    """Fill n rows (row0..row0+n-1) at a device or host-mapped address."""
    rc = _load().synth_rows_gpu(seed, d, row0, n, ctypes.c_void_p(out_ptr),
                                ctypes.c_void_p(stream_ptr))
    if rc != 0:
        raise RuntimeError(f"synth_rows_gpu failed ({rc})")


def decode_inputs(w: Workload):
    """(hist [S, K-1] int32 right-aligned, hist_len [S] int32, new_tok [steps, S] int32)."""
    S, H = w.dec_S, w.K - 1
    hist = np.full((S, H), -1, np.int32)
    hl = np.full(S, min(w.dec_hist, H), np.int32)
    for s in range(S):
        h = int(hl[s])
        if h:
            hist[s, H - h:] = zipf_tokens(w, stream_seed(w, S_DEC_HIST, s), h, inject=False)
    new = np.empty((w.dec_steps, S), np.int32)
    for s in range(S):
        new[:, s] = zipf_tokens(w, stream_seed(w, S_DEC_TOK, s), w.dec_steps, inject=False)
    return hist, hl, new


# ------------------------------------------------------------ f-gram model
@dataclasses.dataclass(frozen=True)
class FgramModel:
    """Shape of the f-gram transformer (A_fgram) whose weights are drawn here.

    The packed weight buffer holds, per layer, four row-major bf16 matrices:
    qkv [3d x d] (query, key, value rows), o [d x d], gu [2 ffw x d] (gate and
    up rows interleaved in groups of 16: rows 32g..32g+15 are the gates of
    features 16g..16g+15, the next 16 rows their ups), down [d x ffw]. With
    absolute positions (the paper's scheme, Appendix F) the buffer ends with
    the position table P [max_pos x d] after the last layer. Every entry is an
    independent draw of the bf16 row generator (std 0.02).
    """
    name: str
    mid: int          # model id, mixed into every seed
    d: int
    n_heads: int
    ffw: int
    n_layers: int
    max_pos: int = 8              # positions of P: the longest f-gram the model takes
    position: str = "absolute"    # "absolute" (P added to the input) or "rotary"

    def shapes(self):
        d, f = self.d, self.ffw
        return (("qkv", 3 * d, d), ("o", d, d), ("gu", 2 * f, d), ("down", d, f))

    @property
    def layer_elems(self) -> int:
        return sum(r * c for _, r, c in self.shapes())

    @property
    def pos_offset(self) -> int:
        """Element offset of P (after the last layer)."""
        return self.n_layers * self.layer_elems

    @property
    def pos_elems(self) -> int:
        return self.max_pos * self.d if self.position == "absolute" else 0

    @property
    def n_elems(self) -> int:
        return self.n_layers * self.layer_elems + self.pos_elems

    def offset(self, layer: int, which: str) -> int:
        off = layer * self.layer_elems
        for name, r, c in self.shapes():
            if name == which:
                return off
            off += r * c
        raise KeyError(which)


MODELS: Dict[str, FgramModel] = {
    # small enough for the fp64 oracle on every f-gram of a test
    "tiny": FgramModel("tiny", 20, 256, 4, 512, 2),
    # the 711M OLMo shape the paper uses for its smaller f-gram model
    # (d_model 2048, ffw 8192, 12 layers; 16 heads of 128); 3 positions, the
    # longest f-gram of the lists it precomputes (K = 3)
    "olmo_711m": FgramModel("olmo_711m", 21, 2048, 16, 8192, 12, max_pos=3),
}


def model_seed(m: FgramModel, layer: int, which: int) -> int:
    return int(_load().synth_stream_seed(MASTER_SEED, m.mid, S_MODEL, layer * 4 + which))


def model_weights_cpu(m: FgramModel) -> np.ndarray:
    """The packed weight buffer as raw bf16 words, [n_elems] uint16."""
    out = np.empty(m.n_elems, np.uint16)
    for layer in range(m.n_layers):
        for k, (name, r, c) in enumerate(m.shapes()):
            off = m.offset(layer, name)
            out[off:off + r * c] = rows_range_cpu(model_seed(m, layer, k), c, 0, r).reshape(-1)
    if m.pos_elems:
        out[m.pos_offset:] = rows_range_cpu(model_seed(m, m.n_layers, 0), m.d, 0,
                                            m.max_pos).reshape(-1)
    return out


def model_weights_gpu(m: FgramModel, out_ptr: int, stream_ptr: int) -> None:
    """The same buffer written at a device address (2 bytes per element)."""
    for layer in range(m.n_layers):
        for k, (name, r, c) in enumerate(m.shapes()):
            rows_gpu(model_seed(m, layer, k), c, 0, r, out_ptr + 2 * m.offset(layer, name),
                     stream_ptr)
    if m.pos_elems:
        rows_gpu(model_seed(m, m.n_layers, 0), m.d, 0, m.max_pos, out_ptr + 2 * m.pos_offset,
                 stream_ptr)
