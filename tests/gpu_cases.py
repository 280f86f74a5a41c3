"""Shared set-up for the GPU tests: seeded workloads on the device and the
oracle's answer for them. Inputs come from ``synth`` only; expected values
come from ``oracle`` only."""

import numpy as np
import torch

import oracle
import synth
import paper_2502_01637_gb300 as scone

DEV = "cuda:0"


def dev_rows(a: np.ndarray) -> torch.Tensor:
    """uint16 rows -> int16 device tensor (raw bf16 bits)."""
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(DEV)


def gpu_rows(seed: int, n: int, d: int) -> torch.Tensor:
    """Seeded rows generated directly on the device (same bytes as synth.rows_cpu)."""
    t = torch.empty((max(n, 1), d), dtype=torch.int16, device=DEV)
    if n:
        synth.rows_gpu(seed, d, 0, n, t.data_ptr(), torch.cuda.current_stream().cuda_stream)
    return t[:n]


class SmallCase:
    """A workload small enough for the oracle to answer every position."""

    def __init__(self, w: synth.Workload, fgrams=None, tok=None):
        self.w = w
        if fgrams is None:
            self.fg_tok, self.fg_len, _ = synth.fgram_set(w)
        else:
            self.fg_tok, self.fg_len = fgrams
        self.tok = synth.query_tokens(w) if tok is None else np.ascontiguousarray(tok, np.int32)
        self.F = synth.rows_cpu(synth.F_seed(w), w.d, np.arange(self.fg_len.shape[0]))
        self.T = synth.rows_cpu(synth.T_seed(w), w.d, np.arange(w.vocab))
        self.oracle = oracle.Oracle(self.fg_tok, self.fg_len, w.K, w.vocab)

    def expected(self):
        return self.oracle.embed(self.tok, self.F, self.T)

    def build(self, F_location=scone.SCONE_ROWS_DEVICE, load_factor=0.0, F=None):
        Fd = dev_rows(self.F) if F is None else F
        return scone.scone_table_build(self.fg_tok, self.fg_len, self.w.K, self.w.vocab, self.w.d,
                                       Fd, dev_rows(self.T), F_location=F_location,
                                       load_factor=load_factor)


def run_embed(table, tok: np.ndarray, d: int, mode: str = "fused", out_offset: int = 0):
    """Runs the path on tok [B, L]; returns (out uint16 [n, d], row int32, len uint8)."""
    t = torch.from_numpy(np.ascontiguousarray(tok, np.int32)).to(DEV)
    n = t.numel()
    buf = torch.empty(n * d + out_offset, dtype=torch.int16, device=DEV)
    out = buf[out_offset:]
    row = torch.empty(n, dtype=torch.int32, device=DEV)
    ln = torch.empty(n, dtype=torch.uint8, device=DEV)
    if mode == "fused":
        scone.scone_embed(table, t, out, row, ln)
    elif mode == "fused_noaux":
        scone.scone_embed(table, t, out)
        scone.scone_match(table, t, row, ln)
    else:
        scone.scone_match(table, t, row, ln)
        scone.scone_embed_gather(table, t.reshape(-1), row, out)
    torch.cuda.synchronize()
    return (out.cpu().numpy().view(np.uint16).reshape(n, d), row.cpu().numpy(),
            ln.cpu().numpy())
