"""SCONE inference-time input embedding on one GB300 (sm_103a).

Thin Python binding over the C ABI in ``include/scone.h`` (``libscone.so``,
built next to this file by ``__graft_entry__.build()``). Every function has
the C name and only marshals arguments: torch tensors become device
addresses, the current CUDA stream is passed through, and every step of the
path runs in the library's kernels. There is no CPU fallback: if the
library is missing or a call fails, an exception is raised.

Tensors carrying bf16 rows may be ``torch.bfloat16`` or ``torch.int16``
(raw bits); token tensors are ``torch.int32``.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libscone.so")

SCONE_OK = 0
SCONE_ERR_INVALID_ARG = -1
SCONE_ERR_TOKEN_RANGE = -2
SCONE_ERR_DUPLICATE_FGRAM = -3
SCONE_ERR_TABLE_FULL = -4
SCONE_ERR_PROBE_LIMIT = -5
SCONE_ERR_UNSUPPORTED = -6
SCONE_ERR_CUDA = -7
SCONE_ERR_NOMEM = -8
SCONE_ROWS_DEVICE = 0
SCONE_ROWS_HOST_MAPPED = 1
SCONE_COPY_AUTO = 0
SCONE_COPY_REGISTERS = 1
SCONE_COPY_BULK = 2
SCONE_COPY_SPLIT = 3
SCONE_COPY_PIPELINED = 4
SCONE_GEMM_STORE = 0
SCONE_GEMM_RESIDUAL = 1
SCONE_GEMM_SWIGLU = 2
SCONE_FGRAM_POS_ABSOLUTE = 0
SCONE_FGRAM_POS_ROTARY = 1

EXPORTS = ("scone_table_build", "scone_table_destroy", "scone_table_rebuild_noalloc",
           "scone_fgram_suffix_index",
           "scone_table_get_info", "scone_table_set_probe_limit", "scone_table_set_copy_mode",
           "scone_match", "scone_prescan", "scone_embed_gather", "scone_embed",
           "scone_decode_create", "scone_decode_step", "scone_decode_get_history",
           "scone_decode_destroy", "scone_status", "scone_host_alloc", "scone_host_free",
           "scone_embed_varlen", "scone_rowstore_open", "scone_rowstore_gather",
           "scone_rowstore_get_stats", "scone_rowstore_close", "scone_rowstore_probe_reads",
           "scone_gemm_bf16",
           "scone_gemm_bf16_variant", "scone_fgram_model_create",
           "scone_fgram_model_destroy", "scone_fgram_precompute", "scone_fgram_discover",
           "scone_discover_create", "scone_discover_destroy", "scone_discover_set_table_slack",
           "scone_strerror", "scone_version")

_lib = None
_vp = ctypes.c_void_p
_i32, _i64 = ctypes.c_int32, ctypes.c_int64


class SconeError(RuntimeError):
    def __init__(self, code: int, what: str):
        msg = load_library().scone_strerror(code).decode()
        super().__init__(f"{what}: {msg} ({code})")
        self.code = code


class scone_table_info(ctypes.Structure):
    _fields_ = [("n_fgrams", _i64), ("n_slots", _i64), ("n_buckets", _i64),
                ("slot_bytes", _i32), ("key_bits", _i32), ("bits_per_token", _i32),
                ("K", _i32), ("vocab", _i32), ("d", _i32), ("F_location", _i32),
                ("max_insert_probe", _i32), ("table_bytes", _i64), ("F_bytes", _i64),
                ("T_bytes", _i64), ("n_markers", _i64), ("suffix_index", _i32)]

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_}


class scone_rowstore_stats(ctypes.Structure):
    _fields_ = [("positions", _i64), ("misses", _i64), ("rows_read", _i64), ("bytes_read", _i64),
                ("direct_io", _i32)]

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_}


class scone_discover_stats(ctypes.Structure):
    _fields_ = [("candidates", _i64 * 9), ("distinct", _i64 * 9), ("frequent", _i64 * 9),
                ("flushes", _i64 * 9), ("threshold", _i64), ("selected_at_threshold", _i64),
                ("table_bytes_max", _i64), ("ms_bin", ctypes.c_double * 9),
                ("ms_count", ctypes.c_double * 9), ("ms_flag", ctypes.c_double * 9),
                ("ms_scan", ctypes.c_double * 9), ("estimate", _i64 * 9),
                ("table_rebuilds", _i64), ("ms_select", ctypes.c_double),
                ("ms_total", ctypes.c_double), ("ms_alloc_host", ctypes.c_double),
                ("workspace_bytes", _i64)]

    def as_dict(self):
        out = {}
        for k, _ in self._fields_:
            v = getattr(self, k)
            out[k] = list(v) if not isinstance(v, (int, float)) else v
        return out


def load_library():
    """Loads libscone.so (raises if it was not built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: run __graft_entry__.build() "
                           "(there is no CPU fallback)")
    lib = ctypes.CDLL(LIB_PATH)
    lib.scone_table_build.argtypes = [_vp, _vp, _i64, _i32, _i32, _i32, _vp, _i32, _vp,
                                      ctypes.c_float, _vp, ctypes.POINTER(_vp)]
    lib.scone_table_destroy.argtypes = [_vp]
    lib.scone_fgram_suffix_index.argtypes = [_vp, _vp, _i64, _i32, _vp, _vp, _vp, _i64,
                                             ctypes.POINTER(_i64)]
    lib.scone_table_rebuild_noalloc.argtypes = [_vp, _vp, _vp, _i64, _vp, _vp]
    lib.scone_table_get_info.argtypes = [_vp, ctypes.POINTER(scone_table_info)]
    lib.scone_table_set_probe_limit.argtypes = [_vp, _i64]
    lib.scone_table_set_copy_mode.argtypes = [_vp, _i32]
    lib.scone_match.argtypes = [_vp, _vp, _i32, _i32, _vp, _vp, _vp]
    lib.scone_prescan.argtypes = [_vp, _vp, _i64, _i32, _vp, _vp, _i64, _vp]
    lib.scone_embed_gather.argtypes = [_vp, _vp, _vp, _i64, _vp, _vp]
    lib.scone_embed.argtypes = [_vp, _vp, _i32, _i32, _vp, _vp, _vp, _vp]
    lib.scone_embed_varlen.argtypes = [_vp, _vp, _i64, _vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp]
    lib.scone_rowstore_open.argtypes = [ctypes.c_char_p, _i64, _i32, _i64, _i32,
                                        ctypes.POINTER(_vp)]
    lib.scone_rowstore_gather.argtypes = [_vp, _vp, _vp, _vp, _i64, _vp, _vp]
    lib.scone_rowstore_get_stats.argtypes = [_vp, ctypes.POINTER(scone_rowstore_stats)]
    lib.scone_rowstore_close.argtypes = [_vp]
    lib.scone_rowstore_probe_reads.argtypes = [_vp, _i64, ctypes.c_uint64,
                                               ctypes.POINTER(ctypes.c_double),
                                               ctypes.POINTER(ctypes.c_double)]
    lib.scone_gemm_bf16.argtypes = [_vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _vp, _vp]
    lib.scone_gemm_bf16_variant.argtypes = [_vp, _vp, _vp, _vp, _i32, _i32, _i32, _i32, _i32,
                                            _vp, _vp]
    lib.scone_fgram_model_create.argtypes = [_i32, _i32, _i32, _i32, _i32, _i32, _vp, _i64,
                                             ctypes.POINTER(_vp)]
    lib.scone_fgram_model_destroy.argtypes = [_vp]
    lib.scone_fgram_precompute.argtypes = [_vp, _vp, _vp, _i64, _i32, _vp, _i32, _vp, _vp]
    lib.scone_decode_create.argtypes = [_vp, _i32, _vp, _vp, ctypes.POINTER(_vp)]
    lib.scone_decode_step.argtypes = [_vp, _vp, _vp, _vp, _vp, _vp]
    lib.scone_decode_get_history.argtypes = [_vp, _vp, _vp]
    lib.scone_decode_destroy.argtypes = [_vp]
    lib.scone_status.argtypes = [_vp, _vp]
    lib.scone_host_alloc.argtypes = [_i64, ctypes.POINTER(_vp)]
    lib.scone_host_free.argtypes = [_vp]
    lib.scone_fgram_discover.argtypes = [_vp, _vp, _i32, _i32, _i32, _i32, _i64, _i32, _vp, _vp,
                                         _vp, ctypes.POINTER(_i64),
                                         ctypes.POINTER(scone_discover_stats), _vp]
    lib.scone_discover_create.argtypes = [ctypes.POINTER(_vp)]
    lib.scone_discover_destroy.argtypes = [_vp]
    lib.scone_discover_set_table_slack.argtypes = [_vp, ctypes.c_double]
    lib.scone_strerror.argtypes = [ctypes.c_int]
    lib.scone_strerror.restype = ctypes.c_char_p
    lib.scone_version.argtypes = []
    for name in EXPORTS:
        if name != "scone_strerror":
            getattr(lib, name).restype = ctypes.c_int
    _lib = lib
    return lib


def _check(rc: int, what: str):
    if rc != SCONE_OK:
        raise SconeError(rc, what)


def _stream(stream) -> int:
    import torch

    if stream is None:
        # the raw handle of the current stream, without building a Stream object
        # (a few microseconds per call, which a decode step feels)
        raw = getattr(torch._C, "_cuda_getCurrentRawStream", None)
        if raw is not None:
            return raw(torch.cuda.current_device())
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _ptr(t) -> Optional[int]:
    """Address of a tensor, numpy array, raw int address, or None."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, HostBuffer):
        return t.ptr
    if isinstance(t, np.ndarray):
        assert t.flags["C_CONTIGUOUS"]
        return t.ctypes.data
    assert t.is_contiguous(), "tensors must be contiguous"
    return t.data_ptr()


class Table:
    """A built f-gram table (owns the C handle; borrows F and T)."""

    def __init__(self, handle: ctypes.c_void_p, keep):
        self._h = handle
        self._keep = keep   # F and T must outlive the table
        self._d = None

    @property
    def d(self) -> int:
        """Row width (elements), read once from the table."""
        if self._d is None:
            self._d = self.info()["d"]
        return self._d

    @property
    def handle(self) -> ctypes.c_void_p:
        if self._h is None:
            raise RuntimeError("table was closed")
        return self._h

    def info(self) -> dict:
        return scone_table_get_info(self)

    def close(self):
        if self._h is not None:
            load_library().scone_table_destroy(self._h)
            self._h = None
            self._keep = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def scone_table_build(fgram_tok: np.ndarray, fgram_len: np.ndarray, K: int, vocab: int, d: int,
                      F, T, F_location: int = SCONE_ROWS_DEVICE, load_factor: float = 0.0,
                      stream=None) -> Table:
    """Builds the f-gram table. fgram_tok host [N, K] int32, fgram_len host [N] uint8.

    F is a device tensor [N, d] (or a host-mapped address when F_location is
    SCONE_ROWS_HOST_MAPPED); T a device tensor [vocab, d].
    """
    lib = load_library()
    ft = np.ascontiguousarray(fgram_tok, dtype=np.int32).reshape(-1)
    fl = np.ascontiguousarray(fgram_len, dtype=np.uint8).reshape(-1)
    n = fl.shape[0]
    if ft.shape[0] != n * K:
        raise ValueError("fgram_tok must be [n_fgrams, K]")
    # T is read for every position without an f-gram; F only by the calls that
    # copy f-gram rows (a table that only selects rows for a row store may hold
    # a one-row placeholder F)
    _need("scone_table_build", ("T", T, 2 * max(vocab, 0) * max(d, 0)))
    h = _vp()
    rc = lib.scone_table_build(_ptr(ft) if n else None, _ptr(fl) if n else None, n, K, vocab, d,
                               _ptr(F), F_location, _ptr(T), load_factor, _stream(stream),
                               ctypes.byref(h))
    _check(rc, "scone_table_build")
    return Table(h, (F, T))


def scone_fgram_suffix_index(fgram_tok: np.ndarray, fgram_len: np.ndarray, K: int):
    """The suffix index scone_table_build gives a table (host only): returns
    (ext [N] uint8, marker_tok [M, K] int32 padded with -1, marker_len [M] uint8)."""
    lib = load_library()
    ft = np.ascontiguousarray(fgram_tok, dtype=np.int32).reshape(-1)
    fl = np.ascontiguousarray(fgram_len, dtype=np.uint8).reshape(-1)
    n = fl.shape[0]
    if ft.shape[0] != n * K:
        raise ValueError("fgram_tok must be [n_fgrams, K]")
    ext = np.zeros(n, np.uint8)
    count = _i64(0)
    args = (_ptr(ft) if n else None, _ptr(fl) if n else None, n, K)
    _check(lib.scone_fgram_suffix_index(*args, _ptr(ext) if n else None, None, None, 0,
                                        ctypes.byref(count)), "scone_fgram_suffix_index")
    m = count.value
    mt = np.full((m, K), -1, np.int32)
    ml = np.zeros(m, np.uint8)
    if m:
        _check(lib.scone_fgram_suffix_index(*args, None, _ptr(mt), _ptr(ml), m,
                                            ctypes.byref(count)), "scone_fgram_suffix_index")
    return ext, mt, ml


def scone_table_destroy(table: Table) -> None:
    table.close()


def scone_table_rebuild_noalloc(table: Table, fgram_tok: np.ndarray, fgram_len: np.ndarray, F,
                                stream=None) -> None:
    """Swaps a new f-gram list (and its rows F) into an existing table without
    allocating: for callers that may not call cudaMalloc at that point (device
    memory owned by another allocator, or threads that must not pay for
    allocation and the device-wide synchronization cudaFree can cause). The
    list must fit the table (at most 0.85 of its slots) and the library's
    fixed device scratch (SCONE_REBUILD_SCRATCH_BYTES); calls that overlap on
    the GPU race on that scratch. Synchronizes the stream.

    Work captured before the call (a CUDA graph of embed or decode launches)
    still holds the old list's F, row count and hash seed: capture it again
    after the call.

    The table keeps referencing the F it reads: the new F after a successful
    call with a non-empty list, the old F after a refused call (the table is
    unchanged then), and both after a CUDA error.
    """
    K = table.info()["K"]
    ft = np.ascontiguousarray(fgram_tok, dtype=np.int32).reshape(-1)
    fl = np.ascontiguousarray(fgram_len, dtype=np.uint8).reshape(-1)
    n = fl.shape[0]
    if ft.shape[0] != n * K:
        raise ValueError("fgram_tok must be [n_fgrams, K]")
    rc = load_library().scone_table_rebuild_noalloc(table.handle, _ptr(ft) if n else None,
                                                    _ptr(fl) if n else None, n, _ptr(F),
                                                    _stream(stream))
    old_F, T = table._keep if table._keep else (None, None)
    if rc == SCONE_OK and n > 0:
        table._keep = (F, T)
    elif rc == SCONE_ERR_CUDA:
        table._keep = ((old_F, F), T)
    _check(rc, "scone_table_rebuild_noalloc")


def scone_table_get_info(table: Table) -> dict:
    info = scone_table_info()
    _check(load_library().scone_table_get_info(table.handle, ctypes.byref(info)),
           "scone_table_get_info")
    return info.as_dict()


def scone_table_set_probe_limit(table: Table, max_buckets: int) -> None:
    _check(load_library().scone_table_set_probe_limit(table.handle, max_buckets),
           "scone_table_set_probe_limit")


def scone_table_set_copy_mode(table: Table, mode: int) -> None:
    _check(load_library().scone_table_set_copy_mode(table.handle, mode),
           "scone_table_set_copy_mode")


def _bl(tok):
    if tok.dim() == 2:
        return tok.shape[0], tok.shape[1]
    return 1, tok.shape[0]


def scone_match(table: Table, tok, row, len=None, stream=None) -> None:
    """tok [B, L] (or [n]) int32 device; row int32 and len uint8 of the same count."""
    B, L = _bl(tok)
    _need("scone_match", ("row", row, 4 * B * L), ("len", len, B * L))
    _check(load_library().scone_match(table.handle, _ptr(tok), B, L, _ptr(row), _ptr(len),
                                      _stream(stream)), "scone_match")


def _nbytes(x) -> Optional[int]:
    """Size in bytes of a buffer argument, or None for a raw address."""
    if x is None or isinstance(x, int):
        return None
    if isinstance(x, HostBuffer):
        return x.nbytes
    if isinstance(x, np.ndarray):
        return x.nbytes
    return x.numel() * x.element_size()


def _need(call: str, *specs) -> None:
    """specs: (name, buffer, bytes the call reads or writes there). A buffer of
    known size that holds fewer bytes raises ValueError before the call, so no
    kernel or copy runs past it; raw addresses and None pass unchecked."""
    for name, buf, need in specs:
        size = _nbytes(buf)
        if size is not None and size < need:
            raise ValueError(f"{call}: {name} holds {size} bytes, needs {need}")


def scone_prescan(table: Table, tok, B: int, L: int, row, len=None, chunk_tokens: int = 0,
                  stream=None) -> None:
    """Tags a corpus in host memory (tok, row, len: host addresses or buffers of
    B * L entries), staged through HBM in chunks of whole sequences; returns
    when the tags are in host memory. Buffers whose size is known are checked
    against B * L entries first (the copies would otherwise run past them)."""
    n = max(B, 0) * max(L, 0)
    _need("scone_prescan", ("tok", tok, 4 * n), ("row", row, 4 * n), ("len", len, n))
    _check(load_library().scone_prescan(table.handle, _ptr(tok), B, L, _ptr(row), _ptr(len),
                                        chunk_tokens, _stream(stream)), "scone_prescan")


def scone_embed_gather(table: Table, tok, row, out, stream=None) -> None:
    n = tok.numel()
    _need("scone_embed_gather", ("row", row, 4 * n), ("out", out, 2 * n * table.d))
    _check(load_library().scone_embed_gather(table.handle, _ptr(tok), _ptr(row), tok.numel(),
                                             _ptr(out), _stream(stream)), "scone_embed_gather")


def _tok_ptr(tok) -> int:
    """Token address for the kernels: a CUDA tensor, or a pinned (page-locked,
    device-mapped) CPU tensor that the kernel reads over the host link."""
    if hasattr(tok, "is_cuda") and not tok.is_cuda and not tok.is_pinned():
        raise ValueError("host tokens must be pinned (tensor.pin_memory()) to be read by "
                         "the device")
    if isinstance(tok, np.ndarray):
        raise ValueError("tokens must be a CUDA or pinned CPU tensor")
    return _ptr(tok)


def scone_embed(table: Table, tok, out, row=None, len=None, stream=None) -> None:
    """Fused Algorithm 1: out [B*L, d] bf16 rows; row / len optional. tok may
    be a pinned CPU tensor: the kernel then reads it over the host link."""
    B, L = _bl(tok)
    n = B * L
    _need("scone_embed", ("out", out, 2 * n * table.d), ("row", row, 4 * n), ("len", len, n))
    _check(load_library().scone_embed(table.handle, _tok_ptr(tok), B, L, _ptr(out), _ptr(row),
                                      _ptr(len), _stream(stream)), "scone_embed")


def scone_embed_varlen(table: Table, tok, cu_seqlens, out, state=None, seq_slot=None, row=None,
                       len=None, stream=None) -> None:
    """Packed ragged batch: tok [n_tok] int32, cu_seqlens [n_seq + 1] int32
    (device); with a DecodeState, sequence b continues slot seq_slot[b] (or
    b) and the slots' histories advance."""
    n_seq = cu_seqlens.numel() - 1
    n = tok.numel()
    _need("scone_embed_varlen", ("out", out, 2 * n * table.d), ("row", row, 4 * n),
          ("len", len, n), ("seq_slot", seq_slot, 4 * max(n_seq, 0)))
    _check(load_library().scone_embed_varlen(
        table.handle, _ptr(tok), tok.numel(), _ptr(cu_seqlens), n_seq,
        state.handle if state is not None else None, _ptr(seq_slot), _ptr(out), _ptr(row),
        _ptr(len), _stream(stream)), "scone_embed_varlen")


def scone_gemm_bf16(A, B, C, R=None, epilogue: int = SCONE_GEMM_STORE, status=None,
                    stream=None, variant: int = 0) -> None:
    """C = epilogue(A B^T) on the tensor cores; A [M, K], B [N, K], C [M, N]
    (or [M, N/2] for SwiGLU), bf16 (or int16 raw bits) device tensors. status:
    a device int32 tensor of one element (allocated here if None; SconeError
    if a pipeline wait timed out)."""
    import torch

    M, K = A.shape
    N = B.shape[0]
    if B.dim() != 2 or B.shape[1] != K:
        raise ValueError(f"scone_gemm_bf16: B must be [N, {K}], got {tuple(B.shape)}")
    c_cols = N // 2 if epilogue == SCONE_GEMM_SWIGLU else N
    _need("scone_gemm_bf16", ("C", C, 2 * M * c_cols),
          ("R", R if epilogue == SCONE_GEMM_RESIDUAL else None, 2 * M * N))
    own = status is None
    if own:
        status = torch.zeros(1, dtype=torch.int32, device=A.device)
    _check(load_library().scone_gemm_bf16_variant(_ptr(A), _ptr(B), _ptr(R), _ptr(C), M, N, K,
                                                   epilogue, variant, _ptr(status),
                                                   _stream(stream)), "scone_gemm_bf16")
    if own:
        code = int(status.item())
        if code:
            raise SconeError(code, "scone_gemm_bf16 (device)")


class FgramModel:
    """The f-gram model on the device (borrows its packed weights). With
    absolute positions (the default) the weights end with P [max_pos, d]."""

    def __init__(self, d: int, n_heads: int, ffw: int, n_layers: int, weights, batch: int = 0,
                 max_pos: int = 8, position: int = SCONE_FGRAM_POS_ABSOLUTE):
        h = _vp()
        _check(load_library().scone_fgram_model_create(d, n_heads, ffw, n_layers, max_pos,
                                                       position, _ptr(weights), batch,
                                                       ctypes.byref(h)),
               "scone_fgram_model_create")
        self._h = h
        self._keep = weights
        self.d = d

    @property
    def handle(self):
        if self._h is None:
            raise RuntimeError("model was closed")
        return self._h

    def close(self):
        if self._h is not None:
            load_library().scone_fgram_model_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def scone_fgram_model_create(d, n_heads, ffw, n_layers, max_pos, position, weights,
                             batch=0) -> FgramModel:
    return FgramModel(d, n_heads, ffw, n_layers, weights, batch, max_pos, position)


def scone_fgram_model_destroy(model: FgramModel) -> None:
    model.close()


def scone_fgram_precompute(model: FgramModel, fgram_tok, fgram_len, T, F,
                           vocab: Optional[int] = None, stream=None) -> None:
    """F rows of the f-grams: fgram_tok [n, K] int32 and fgram_len [n] uint8 device
    tensors, T [vocab, d] device, F [n, d] device tensor (or host-mapped address)."""
    n, K = fgram_tok.shape
    vocab = T.shape[0] if vocab is None else vocab
    d = model.d
    _need("scone_fgram_precompute", ("fgram_len", fgram_len, n), ("T", T, 2 * vocab * d),
          ("F", F, 2 * n * d))
    _check(load_library().scone_fgram_precompute(model.handle, _ptr(fgram_tok), _ptr(fgram_len), n,
                                                 K, _ptr(T), vocab, _ptr(F), _stream(stream)),
           "scone_fgram_precompute")


class RowStore:
    """F in a file with an HBM row cache (scone_rowstore_*)."""

    def __init__(self, path: str, n_rows: int, d: int, cache_rows: int, threads: int = 0):
        h = _vp()
        _check(load_library().scone_rowstore_open(os.fsencode(path), n_rows, d, cache_rows,
                                                  threads, ctypes.byref(h)),
               "scone_rowstore_open")
        self._h = h

    @property
    def handle(self):
        if self._h is None:
            raise RuntimeError("row store was closed")
        return self._h

    def stats(self) -> dict:
        st = scone_rowstore_stats()
        _check(load_library().scone_rowstore_get_stats(self.handle, ctypes.byref(st)),
               "scone_rowstore_get_stats")
        return st.as_dict()

    def close(self):
        if self._h is not None:
            load_library().scone_rowstore_close(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def scone_rowstore_open(path, n_rows, d, cache_rows, threads=0) -> RowStore:
    return RowStore(path, n_rows, d, cache_rows, threads)


def scone_rowstore_close(store: RowStore) -> None:
    store.close()


def scone_rowstore_get_stats(store: RowStore) -> dict:
    return store.stats()


def scone_rowstore_probe_reads(store: RowStore, n_reads: int, seed: int = 1) -> dict:
    """Random-row read rate of the store's file with its own threads and I/O mode."""
    rows, nbytes = ctypes.c_double(), ctypes.c_double()
    _check(load_library().scone_rowstore_probe_reads(store.handle, n_reads, seed,
                                                     ctypes.byref(rows), ctypes.byref(nbytes)),
           "scone_rowstore_probe_reads")
    return {"rows_per_s": rows.value, "bytes_per_s": nbytes.value}


def scone_rowstore_gather(store: RowStore, table: Table, tok, row, out, stream=None) -> None:
    """out[t] = F[row[t]] from the store (or T[tok[t]] where row[t] < 0)."""
    n = row.numel()
    _need("scone_rowstore_gather", ("tok", tok, 4 * n), ("out", out, 2 * n * table.d))
    _check(load_library().scone_rowstore_gather(store.handle, table.handle, _ptr(tok), _ptr(row),
                                                row.numel(), _ptr(out), _stream(stream)),
           "scone_rowstore_gather")


class DecodeState:
    def __init__(self, handle, table: Table, S: int, H: int):
        self._h = handle
        self._table = table
        self.S, self.H = S, H

    @property
    def handle(self):
        if self._h is None:
            raise RuntimeError("decode state was closed")
        return self._h

    def close(self):
        if self._h is not None:
            load_library().scone_decode_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def scone_decode_create(table: Table, hist: np.ndarray, hist_len: np.ndarray) -> DecodeState:
    """hist host [S, K-1] int32 right-aligned; hist_len host [S] int32 in [0, K-1]."""
    hist = np.ascontiguousarray(hist, dtype=np.int32)
    hl = np.ascontiguousarray(hist_len, dtype=np.int32)
    S = hl.shape[0]
    h = _vp()
    _check(load_library().scone_decode_create(table.handle, S, _ptr(hist), _ptr(hl),
                                              ctypes.byref(h)), "scone_decode_create")
    return DecodeState(h, table, S, hist.shape[1] if hist.ndim == 2 else 0)


def scone_decode_step(state: DecodeState, new_tok, out, row=None, len=None, stream=None) -> None:
    """One decode step; new_tok [S] int32, a CUDA tensor or a pinned CPU tensor
    (read by the kernel over the host link)."""
    S = state.S
    _need("scone_decode_step", ("new_tok", new_tok, 4 * S),
          ("out", out, 2 * S * state._table.d if out is not None else 0),
          ("row", row, 4 * S), ("len", len, S))
    _check(load_library().scone_decode_step(state.handle, _tok_ptr(new_tok), _ptr(out),
                                            _ptr(row), _ptr(len), _stream(stream)),
           "scone_decode_step")


def scone_decode_get_history(state: DecodeState):
    hist = np.empty((state.S, state.H), np.int32)
    hl = np.empty(state.S, np.int32)
    _check(load_library().scone_decode_get_history(state.handle, _ptr(hist), _ptr(hl)),
           "scone_decode_get_history")
    return hist, hl


def scone_decode_destroy(state: DecodeState) -> None:
    state.close()


def scone_status(table: Table, stream=None, raise_on_error: bool = True) -> int:
    """Synchronizes the stream; returns (or raises) the sticky device error."""
    rc = load_library().scone_status(table.handle, _stream(stream))
    if raise_on_error:
        _check(rc, "device status")
    return rc


class HostBuffer:
    """Pinned, device-mapped host memory from scone_host_alloc (for an offloaded F)."""

    def __init__(self, nbytes: int):
        p = _vp()
        _check(load_library().scone_host_alloc(nbytes, ctypes.byref(p)), "scone_host_alloc")
        self.ptr = p.value
        self.nbytes = nbytes

    def numpy(self, dtype=np.uint16) -> np.ndarray:
        """Host view of the buffer (no copy)."""
        buf = (ctypes.c_char * self.nbytes).from_address(self.ptr)
        return np.frombuffer(buf, dtype=dtype)

    def free(self):
        if self.ptr:
            load_library().scone_host_free(self.ptr)
            self.ptr = 0

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def scone_host_alloc(nbytes: int) -> HostBuffer:
    return HostBuffer(nbytes)


def scone_host_free(buf: HostBuffer) -> None:
    buf.free()


class DiscoverWorkspace:
    """Reusable device buffers of scone_fgram_discover (freed by close)."""

    def __init__(self):
        h = _vp()
        _check(load_library().scone_discover_create(ctypes.byref(h)), "scone_discover_create")
        self._h = h

    @property
    def handle(self):
        if self._h is None:
            raise RuntimeError("workspace was closed")
        return self._h

    def set_table_slack(self, slots_per_key: float):
        """Counting-table slots per estimated distinct n-gram (default 4)."""
        _check(load_library().scone_discover_set_table_slack(self.handle, float(slots_per_key)),
               "scone_discover_set_table_slack")

    def close(self):
        if self._h is not None:
            load_library().scone_discover_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def scone_discover_create() -> DiscoverWorkspace:
    return DiscoverWorkspace()


def scone_discover_destroy(ws: DiscoverWorkspace) -> None:
    ws.close()


def scone_fgram_discover(tok, vocab: int, K: int, S: int, min_count: int = 5,
                         fgram_tok=None, fgram_len=None, fgram_count=None,
                         workspace: Optional[DiscoverWorkspace] = None, stream=None):
    """Algorithm 3 by the K-1 counting scans of Sec. 3.2 over a corpus tok
    [B, L] int32 (device tensor, or a HostBuffer address with shape given as
    a (ptr, B, L) tuple). Returns (fgram_tok [n, K] int32, fgram_len [n] uint8,
    fgram_count [n] int32, stats dict); the outputs are device tensors
    (allocated here unless given, each with room for S f-grams). With a
    workspace, repeated calls reuse its device buffers."""
    import torch

    if isinstance(tok, tuple):
        ptr, B, L = tok
        dev = torch.device("cuda", torch.cuda.current_device())
    else:
        B, L = _bl(tok)
        ptr = _ptr(tok)
        dev = tok.device
    if fgram_tok is None:
        fgram_tok = torch.empty((max(S, 1), K), dtype=torch.int32, device=dev)
    if fgram_len is None:
        fgram_len = torch.empty(max(S, 1), dtype=torch.uint8, device=dev)
    if fgram_count is None:
        fgram_count = torch.empty(max(S, 1), dtype=torch.int32, device=dev)
    n_out = _i64()
    st = scone_discover_stats()
    ws = workspace.handle if workspace is not None else None
    _check(load_library().scone_fgram_discover(ws, ptr, B, L, vocab, K, S, min_count,
                                               _ptr(fgram_tok), _ptr(fgram_len),
                                               _ptr(fgram_count), ctypes.byref(n_out),
                                               ctypes.byref(st), _stream(stream)),
           "scone_fgram_discover")
    n = n_out.value
    return fgram_tok[:n], fgram_len[:n], fgram_count[:n], st.as_dict()


def scone_strerror(code: int) -> str:
    return load_library().scone_strerror(code).decode()


def scone_version() -> int:
    return load_library().scone_version()
