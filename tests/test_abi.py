"""The C ABI library loads and exports what include/scone.h declares (CPU).

Also checks the host-side argument validation, which returns before any
CUDA call, so it runs without a GPU.
"""

import ctypes
import os
import re
import subprocess

import numpy as np

import paper_2502_01637_gb300 as scone

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "scone.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(scone_[a-z_0-9]+)\s*\(", src)))


def test_every_declared_symbol_is_exported():
    lib = scone.load_library()
    names = declared_functions()
    assert len(names) >= 14
    for n in names:
        assert hasattr(lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", scone.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (scone_[a-z_0-9]+)", out))
    assert set(names) <= exported, set(names) - exported
    assert set(scone.EXPORTS) == set(names)


def test_strerror_and_version():
    assert scone.scone_strerror(0) == "ok"
    assert "duplicate" in scone.scone_strerror(scone.SCONE_ERR_DUPLICATE_FGRAM)
    assert scone.scone_strerror(-99) == "unknown error"
    assert scone.scone_version() >> 16 == 1


def _build_rc(fgram_tok, fgram_len, K, vocab, d=8, T=0x1000, F=0x2000, lf=0.0, loc=0):
    lib = scone.load_library()
    ft = np.ascontiguousarray(fgram_tok, dtype=np.int32).reshape(-1)
    fl = np.ascontiguousarray(fgram_len, dtype=np.uint8).reshape(-1)
    h = ctypes.c_void_p()
    return lib.scone_table_build(ft.ctypes.data if fl.size else None,
                                 fl.ctypes.data if fl.size else None, fl.size, K, vocab, d, F, loc,
                                 T, lf, None, ctypes.byref(h))


def test_host_validation_returns_before_device_work():
    ok_tok = np.array([[1, 2, -1]], np.int32)
    ok_len = np.array([2], np.uint8)
    inv = scone.SCONE_ERR_INVALID_ARG
    assert _build_rc(ok_tok, ok_len, 1, 10) == inv          # K < 2
    assert _build_rc(ok_tok, ok_len, 9, 10) == inv          # K > 8
    assert _build_rc(ok_tok, ok_len, 3, 0) == inv           # empty vocab
    assert _build_rc(ok_tok, ok_len, 3, 10, d=0) == inv     # d < 1
    assert _build_rc(ok_tok, ok_len, 3, 10, T=0) == inv     # no T
    assert _build_rc(ok_tok, ok_len, 3, 10, F=0) == inv     # no F with f-grams
    assert _build_rc(ok_tok, ok_len, 3, 10, lf=0.99) == inv  # load factor too high
    assert _build_rc(ok_tok, ok_len, 3, 10, lf=0.9) == inv   # above the cuckoo bound 0.85
    assert _build_rc(ok_tok, ok_len, 3, 10, lf=-1.0) == inv
    assert _build_rc(ok_tok, ok_len, 3, 10, loc=7) == inv   # unknown F location
    assert _build_rc(ok_tok, np.array([1], np.uint8), 3, 10) == inv   # 1-gram
    assert _build_rc(ok_tok, np.array([4], np.uint8), 3, 10) == inv   # longer than K
    assert _build_rc(np.array([[1, 10, -1]], np.int32), ok_len, 3, 10) == inv  # token range
    assert _build_rc(np.array([[-1, 2, -1]], np.int32), ok_len, 3, 10) == inv
    # key does not fit: K=8 tokens of 30 bits
    assert _build_rc(np.zeros((1, 8), np.int32), ok_len, 8, 1 << 30) == scone.SCONE_ERR_UNSUPPORTED
    lib = scone.load_library()
    assert lib.scone_table_build(None, None, 0, 3, 10, 8, None, 0, 0x1000, 0.0, None,
                                 None) == inv               # no out pointer


def test_null_handles_rejected():
    lib = scone.load_library()
    inv = scone.SCONE_ERR_INVALID_ARG
    assert lib.scone_match(None, None, 1, 1, None, None, None) == inv
    assert lib.scone_embed(None, None, 1, 1, None, None, None, None) == inv
    assert lib.scone_embed_gather(None, None, None, 1, None, None) == inv
    assert lib.scone_decode_step(None, None, None, None, None, None) == inv
    assert lib.scone_decode_create(None, 1, None, None, None) == inv
    assert lib.scone_status(None, None) == inv
    assert lib.scone_table_destroy(None) == 0
    assert lib.scone_decode_destroy(None) == 0
    assert lib.scone_table_get_info(None, None) == inv
    assert lib.scone_table_set_probe_limit(None, 1) == inv
    assert lib.scone_embed_varlen(None, None, 0, None, 0, None, None, None, None, None,
                                  None) == inv
    assert lib.scone_fgram_discover(None, None, 1, 1, 10, 1, 5, 1, None, None, None, None, None,
                                    None) == inv             # no n_out
    assert lib.scone_discover_create(None) == inv
    assert lib.scone_discover_destroy(None) == 0
    assert lib.scone_discover_set_table_slack(None, 2.5) == inv
    assert lib.scone_prescan(None, None, 1, 1, None, None, 0, None) == inv
    n_markers = ctypes.c_int64(-1)
    assert lib.scone_fgram_suffix_index(None, None, 1, 3, None, None, None, 0,
                                        ctypes.byref(n_markers)) == inv    # list missing
    assert lib.scone_fgram_suffix_index(None, None, 0, 3, None, None, None, 0,
                                        None) == inv                      # no count pointer
    assert lib.scone_fgram_suffix_index(None, None, 0, 3, None, None, None, 0,
                                        ctypes.byref(n_markers)) == 0 and n_markers.value == 0


def test_key_format_boundaries():
    """FMT16 up to K*b = 92, FMT32 up to 220 (K*b + 4 length bits)."""
    # bits per token = ceil(log2 vocab): vocab 2^18 -> 18 bits; K=5 -> 90 <= 92 fits the
    # 16-byte slot; vocab 2^18+1 -> 19 bits -> 95 > 92 needs the 32-byte slot; both are
    # accepted by the host checks (they fail later only because T is not device memory).
    for vocab in (1 << 18, (1 << 18) + 1):
        rc = _build_rc(np.zeros((1, 5), np.int32), np.array([2], np.uint8), 5, vocab)
        assert rc == scone.SCONE_ERR_INVALID_ARG     # T=0x1000 is not device memory
    rc = _build_rc(np.zeros((1, 8), np.int32), np.array([2], np.uint8), 8, 1 << 27)
    assert rc == scone.SCONE_ERR_INVALID_ARG         # 8*27 = 216 <= 220: format fits
    rc = _build_rc(np.zeros((1, 8), np.int32), np.array([2], np.uint8), 8, (1 << 27) + 1)
    assert rc == scone.SCONE_ERR_UNSUPPORTED         # 8*28 = 224 > 220


def test_host_tokens_must_be_pinned():
    """Tokens the kernels read from host memory must be page-locked: the
    binding refuses pageable CPU tensors and numpy arrays before any launch."""
    import numpy as np
    import pytest
    import torch

    import paper_2502_01637_gb300 as scone

    with pytest.raises(ValueError):
        scone._tok_ptr(torch.zeros(8, dtype=torch.int32))
    with pytest.raises(ValueError):
        scone._tok_ptr(np.zeros(8, np.int32))


def test_prescan_buffers_checked_against_the_corpus_size():
    """scone_prescan's wrapper refuses host buffers shorter than B * L entries
    (4 bytes for tokens and rows, 1 for lengths) before the library is
    called, so no copy can run past them."""
    import numpy as np
    import pytest

    import paper_2502_01637_gb300 as scone

    B, L = 3, 5
    ok_tok, ok_row, ok_len = (np.zeros(B * L, np.int32), np.zeros(B * L, np.int32),
                              np.zeros(B * L, np.uint8))
    short = (np.zeros(B * L - 1, np.int32), np.zeros(B * L - 1, np.int32),
             np.zeros(B * L - 1, np.uint8))
    for k, name in enumerate(("tok", "row", "len")):
        args = [ok_tok, ok_row, ok_len]
        args[k] = short[k]
        with pytest.raises(ValueError, match=name):
            scone.scone_prescan(None, args[0], B, L, args[1], args[2])
    assert scone._nbytes(ok_len) == B * L and scone._nbytes(0x1000) is None


def test_output_buffers_checked_against_the_batch():
    """The embed, match, gather, ragged-batch and decode wrappers refuse an
    output (or index) buffer smaller than the batch needs before the library
    is called: the kernels cannot see a tensor's size and would write past
    it. Checked with host tensors and stand-in handles (no device needed)."""
    import types

    import numpy as np
    import pytest
    import torch

    import paper_2502_01637_gb300 as scone

    d, B, L = 16, 2, 3
    n = B * L
    table = types.SimpleNamespace(d=d, handle=None)
    tok = torch.zeros((B, L), dtype=torch.int32)
    out_ok = torch.zeros((n, d), dtype=torch.int16)
    out_short = torch.zeros((n - 1, d), dtype=torch.int16)
    row_short = torch.zeros(n - 1, dtype=torch.int32)
    len_short = torch.zeros(n - 1, dtype=torch.uint8)
    with pytest.raises(ValueError, match="out"):
        scone.scone_embed(table, tok, out_short)
    with pytest.raises(ValueError, match="row"):
        scone.scone_embed(table, tok, out_ok, row=row_short)
    with pytest.raises(ValueError, match="len"):
        scone.scone_embed(table, tok, out_ok, len=len_short)
    with pytest.raises(ValueError, match="row"):
        scone.scone_match(table, tok, row_short)
    with pytest.raises(ValueError, match="out"):
        scone.scone_embed_gather(table, tok.reshape(-1), torch.zeros(n, dtype=torch.int32),
                                 out_short)
    cu = torch.tensor([0, 4, n], dtype=torch.int32)
    with pytest.raises(ValueError, match="out"):
        scone.scone_embed_varlen(table, tok.reshape(-1), cu, out_short)
    with pytest.raises(ValueError, match="seq_slot"):
        scone.scone_embed_varlen(table, tok.reshape(-1), cu, out_ok,
                                 seq_slot=torch.zeros(1, dtype=torch.int32))
    state = types.SimpleNamespace(S=4, _table=table, handle=None)
    with pytest.raises(ValueError, match="out"):
        scone.scone_decode_step(state, torch.zeros(4, dtype=torch.int32), out_short[:3])
    with pytest.raises(ValueError, match="new_tok"):
        scone.scone_decode_step(state, np.zeros(3, np.int32), None)
    # a buffer of the right size passes the check (and then meets the host-token
    # rule: pageable CPU tokens are refused)
    with pytest.raises(ValueError, match="pinned"):
        scone.scone_embed(table, tok, out_ok)


def test_table_build_checks_T_against_the_vocabulary():
    """scone_table_build's wrapper refuses a token table T smaller than vocab
    rows of d bf16 before the library is called (the kernels read T[token]
    for every position without an f-gram)."""
    import numpy as np
    import pytest
    import torch

    import paper_2502_01637_gb300 as scone

    ft = np.array([[1, 2]], np.int32)
    fl = np.array([2], np.uint8)
    T_short = torch.zeros((9, 8), dtype=torch.int16)
    with pytest.raises(ValueError, match="T"):
        scone.scone_table_build(ft, fl, 2, 10, 8, None, T_short)


def test_gemm_and_precompute_buffers_checked():
    """scone_gemm_bf16 refuses B of another K and a C (or R) smaller than the
    epilogue writes (reads); scone_fgram_precompute refuses an F smaller than
    n rows of d. Both before the library is called."""
    import types

    import pytest
    import torch

    import paper_2502_01637_gb300 as scone

    A = torch.zeros((128, 64), dtype=torch.int16)
    with pytest.raises(ValueError, match="B must be"):
        scone.scone_gemm_bf16(A, torch.zeros((256, 32), dtype=torch.int16),
                              torch.zeros((128, 256), dtype=torch.int16))
    B = torch.zeros((256, 64), dtype=torch.int16)
    with pytest.raises(ValueError, match="C"):
        scone.scone_gemm_bf16(A, B, torch.zeros((128, 128), dtype=torch.int16))
    with pytest.raises(ValueError, match="R"):
        scone.scone_gemm_bf16(A, B, torch.zeros((128, 256), dtype=torch.int16),
                              R=torch.zeros((127, 256), dtype=torch.int16),
                              epilogue=scone.SCONE_GEMM_RESIDUAL)
    model = types.SimpleNamespace(d=256, handle=None)
    tok = torch.zeros((4, 3), dtype=torch.int32)
    ln = torch.full((4,), 3, dtype=torch.uint8)
    T = torch.zeros((10, 256), dtype=torch.int16)
    with pytest.raises(ValueError, match="F"):
        scone.scone_fgram_precompute(model, tok, ln, T, torch.zeros((3, 256), dtype=torch.int16))
