"""Throughput of the SCONE inference-time embedding path on one GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl scone|reference]
                    [--workload prefill_1b|large_hbm|stress_k5|tiny|offload_decode]

One step is one pass of the whole path (match + gather, fused in one launch)
over one batch of the workload's seeded synthetic tokens; the default
workload is the largest configuration that fits one GPU, the large
HBM-resident table (64 x 4096 tokens, 1e7 f-grams (41 GB of F), K = 3,
d = 2048, Zipf(1.1) over a 100k vocabulary). Steps rotate over 4 distinct
batches and L2 is flushed (256 MB written, then read) between timed steps;
each step is timed with CUDA events on its stream. Prints one JSON line (see
the keys below). Without --workload, the same process also measures the
1B-model prefill (32 x 2048 tokens, 1e6 f-grams) and the offloaded decode
tier (2e7 f-grams, 82 GB of F in host memory read over the host link, 512
sequences x 256 steps) and reports them under "extra" with their own
roofline, clocks and e2e. ``--impl reference`` times the CPU oracle (the
plain statement of Algorithm 1) on the host cores instead.

Under torchrun (N > 1) every rank embeds its own batches (independent
sequences; weak scaling, no collective on the data path); rank 0 prints the
whole-job throughput over the slowest rank's time.
"""

from __future__ import annotations

import argparse
import ctypes
import glob
import hashlib
import json
import os
import re
import statistics
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "embedded tokens/s at 1 GB300; achieved GB/s vs HBM or host-link roofline"
METRIC_DISCOVER = "corpus tokens/s of f-gram discovery (Algorithm 3, K-1 counting scans) at 1 GB300"


def workload(name):
    import synth

    if name == "prefill_profile":
        # the prefill law at a size an ncu capture handles (about 1.5 GB on the device)
        return synth.WORKLOADS["prefill_1b"].scaled("prefill_profile", B=16,
                                                    quotas=((2, 120000), (3, 80000)))
    if name == "discover_profile":
        # the discover law at a size a full-section ncu capture handles: 2^24
        # corpus tokens (a 0.5 GB counting table, larger than L2)
        return synth.WORKLOADS["discover"].scaled("discover_profile", B=8192,
                                                  quotas=((2, 150_000), (3, 100_000)))
    if name == "decode_profile":
        # the offloaded-decode law with 2e6 f-grams (8 GB of host rows) for ncu captures
        return synth.WORKLOADS["offload_decode"].scaled(
            "decode_profile", quotas=((2, 1_200_000), (3, 800_000)))
    if name == "large_hbm_profile":
        # large_hbm's law (K = 3, d = 2048, Zipf(1.1), 64 x 4096 batches cut to 16) with
        # 7.5e5 f-grams: F 3.1 GB + T 0.4 GB on the device, for counter captures
        return synth.WORKLOADS["large_hbm"].scaled("large_hbm_profile", B=16,
                                                   quotas=((2, 450_000), (3, 300_000)))
    if name == "stress_profile":
        # stress_k5's law (K = 5, d = 1536, phrases injected) with 8 x 8192 tokens and
        # 1e6 f-grams in the same length split: F 3.1 GB + T 0.3 GB on the device
        return synth.WORKLOADS["stress_k5"].scaled(
            "stress_profile", B=8, quotas=((2, 333_333), (3, 333_333), (4, 166_667),
                                           (5, 166_667)))
    if name == "offload_decode_first_seen":
        # the offloaded decode with F's rows in first-seen order instead of by count
        return synth.WORKLOADS["offload_decode"].scaled("offload_decode_first_seen",
                                                        row_order="first_seen")
    return synth.WORKLOADS[name]


N_BATCHES = 4
FLUSH_BYTES = 256 << 20
# the largest configuration that fits one GPU (41 GB of F in HBM)
DEFAULT_WORKLOAD = "large_hbm"


def flush_l2(buf):
    """Writes then reads a buffer twice the size of L2: the previous step's
    lines are gone and the write-backs of the flush itself happen here, not
    inside the next timed kernel."""
    buf.zero_()
    buf.sum()


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """Samples SM clock and throttle reasons through NVML (read-only) in a
    background thread while the timed region runs."""

    REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
               0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
               0x100: "display_clock_setting"}

    def __init__(self, index: int, period_s: float = 0.001):
        self.ok = False
        self.samples = []
        self.reasons = 0
        self.period = period_s
        self._stop = threading.Event()
        try:
            self.nvml = ctypes.CDLL("libnvidia-ml.so.1")
            if self.nvml.nvmlInit_v2() != 0:
                return
            self.h = ctypes.c_void_p()
            if self.nvml.nvmlDeviceGetHandleByIndex_v2(index, ctypes.byref(self.h)) != 0:
                return
            mx = ctypes.c_uint()
            self.nvml.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(mx))   # 1 = SM
            self.max_mhz = mx.value
            self.ok = True
        except OSError:
            pass

    def sample(self):
        if not self.ok:
            return
        c = ctypes.c_uint()
        r = ctypes.c_ulonglong()
        self.nvml.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(c))
        self.nvml.nvmlDeviceGetCurrentClocksEventReasons(self.h, ctypes.byref(r))
        self.samples.append(c.value)
        self.reasons |= r.value

    def _run(self):
        while not self._stop.is_set():
            self.sample()
            time.sleep(self.period)

    def __enter__(self):
        self.sample()
        self._t = threading.Thread(target=self._run, daemon=True)
        self._t.start()
        return self

    def __exit__(self, *a):
        self._stop.set()
        self._t.join()
        self.sample()

    def summary(self):
        if not self.ok or not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvml unavailable"]}
        names = [n for b, n in self.REASONS.items() if self.reasons & b and n != "gpu_idle"]
        return {"sm_mhz": statistics.median(self.samples), "sm_max_mhz": self.max_mhz,
                "reasons": names, "samples": len(self.samples)}


# ------------------------------------------------------------------ helpers
def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


EMBED_SOURCES = ("scone_embed.cu", "scone_device.cuh", "scone_host.h")
PIPE_SOURCES = ("scone_pipe.cu", "scone_walk.cuh", "scone_embed.cu", "scone_device.cuh",
                "scone_host.h")
DISCOVER_SOURCES = ("scone_discover.cu", "scone_device.cuh", "scone_host.h")
VARLEN_SOURCES = ("scone_varlen.cu", "scone_walk.cuh", "scone_device.cuh", "scone_host.h")


def kernel_source_hash(files=EMBED_SOURCES) -> str:
    """Hash of the code (comments and whitespace removed) of the sources that
    compile into a profiled kernel (default: the fused prefill kernel)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2502_01637_gb300", "csrc")
    for f in (os.path.join(csrc, name) for name in files):
        code = re.sub(r"/\*.*?\*/", " ", open(f).read(), flags=re.S)
        code = re.sub(r"//[^\n]*", " ", code)
        h.update(" ".join(code.split()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str, kernel: str = "embed_kernel", files=EMBED_SOURCES,
                     with_note: bool = False):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current kernel sources; else None. With ``with_note``, also the
    summary's one-line note on how the figure was obtained (a capture of a
    smaller case scaled to a full launch, for instance)."""
    p = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.md")
    if not os.path.exists(p):
        return (None, None) if with_note else None
    txt = open(p).read()
    m = re.search(r"dram_bytes_per_launch:\s*(\d+)", txt)
    s = re.search(r"kernel_source_sha256:\s*([0-9a-f]+)", txt)
    n = re.search(r"traffic_note:\s*([^\n]+)", txt)
    ok = bool(m and s and s.group(1) == kernel_source_hash(files))
    val = int(m.group(1)) if ok else None
    if with_note:
        return val, (n.group(1).strip() if (ok and n) else None)
    return val


def algorithmic_bytes_per_token(K: int, d: int) -> int:
    """token id + one 32-byte bucket per probed length + source row + output row."""
    return 4 + 32 * (K - 1) + 4 * d


def dist_setup():
    import torch

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist

        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist

    t = torch.tensor([x], dtype=torch.float64,
                     device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------- scone prefill
def bench_prefill(args, world, rank, local):
    import torch

    import synth
    import paper_2502_01637_gb300 as scone

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = workload(args.workload)
    if getattr(args, "load_factor", None):
        w = w.scaled(w.name, load_factor=args.load_factor)
    n_tok = w.B * w.L
    t0 = time.time()
    fg_tok, fg_len, used = synth.fgram_set(w)
    # rank r embeds sequences of its own sub-streams
    batches_np = [synth.query_tokens(w, range((rank * N_BATCHES + k) * w.B,
                                              (rank * N_BATCHES + k + 1) * w.B))
                  for k in range(N_BATCHES)]
    stream = torch.cuda.current_stream()
    F = torch.empty((w.n_fgrams, w.d), dtype=torch.int16, device=dev)
    T = torch.empty((w.vocab, w.d), dtype=torch.int16, device=dev)
    synth.rows_gpu(synth.F_seed(w), w.d, 0, w.n_fgrams, F.data_ptr(), stream.cuda_stream)
    synth.rows_gpu(synth.T_seed(w), w.d, 0, w.vocab, T.data_ptr(), stream.cuda_stream)
    table = scone.scone_table_build(fg_tok, fg_len, w.K, w.vocab, w.d, F, T,
                                    load_factor=w.load_factor)
    scone.scone_table_set_copy_mode(table, {"auto": scone.SCONE_COPY_AUTO,
                                            "registers": scone.SCONE_COPY_REGISTERS,
                                            "bulk": scone.SCONE_COPY_BULK,
                                            "split": scone.SCONE_COPY_SPLIT,
                                            "pipelined": scone.SCONE_COPY_PIPELINED}[args.copy])
    info = table.info()
    setup_s = time.time() - t0
    batches = [torch.from_numpy(b).to(dev) for b in batches_np]
    out = torch.empty((n_tok, w.d), dtype=torch.int16, device=dev)
    row = torch.empty(n_tok, dtype=torch.int32, device=dev)
    ln = torch.empty(n_tok, dtype=torch.uint8, device=dev)
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    # match statistics of the workload (diagnostic; untimed)
    scone.scone_match(table, batches[0], row, ln)
    hist = torch.bincount(ln.to(torch.int64), minlength=w.K + 1).cpu().numpy()
    scone.scone_status(table)

    def step(k):
        scone.scone_embed(table, batches[k % N_BATCHES], out)

    for k in range(args.warmup):
        flush_l2(flush)
        step(k)
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize()
    wall0 = time.perf_counter()
    with clocks:
        for k in range(args.steps):
            flush_l2(flush)
            ev[k][0].record(stream)
            step(k)
            ev[k][1].record(stream)
        torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    barrier(world)
    scone.scone_status(table)
    per_step_ms = [a.elapsed_time(b) for a, b in ev]
    kernel_ms = sum(per_step_ms) / len(per_step_ms)
    ms_step = max_over_ranks(kernel_ms, world)

    # end to end through the public API with host buffers: pinned tokens in,
    # status word out, the transfers and the sync inside the timed region. The
    # headline passes the pinned tokens to scone_embed, whose kernel reads them
    # over the host link (262 KB per step); "staged" copies them to the device
    # with cudaMemcpyAsync first.
    host_tok = [torch.from_numpy(b).pin_memory() for b in batches_np]
    dev_tok = torch.empty_like(batches[0])
    e2e_steps = max(3, min(args.steps, 50))

    raw_stream = stream.cuda_stream    # the caller's stream handle, passed to each call

    def e2e_step(k, staged):
        if staged:
            dev_tok.copy_(host_tok[k % N_BATCHES], non_blocking=True)
            scone.scone_embed(table, dev_tok, out, stream=raw_stream)
        else:
            scone.scone_embed(table, host_tok[k % N_BATCHES], out, stream=raw_stream)
        scone.scone_status(table, raw_stream)   # syncs the stream, reads the status word

    e2e_ms = {}
    for staged in (False, True):
        for k in range(3):
            e2e_step(k, staged)
        barrier(world)
        e2e_t = []
        for k in range(e2e_steps):
            flush_l2(flush)
            torch.cuda.synchronize()
            t1 = time.perf_counter()
            e2e_step(k, staged)
            e2e_t.append(time.perf_counter() - t1)
        e2e_ms[staged] = max_over_ranks(1e3 * statistics.mean(e2e_t), world)

    per_tok = algorithmic_bytes_per_token(w.K, w.d)
    bytes_launch = per_tok * n_tok
    hbm, peak_src = measured_peaks()
    achieved = bytes_launch / (kernel_ms * 1e-3) / 1e9
    kname_full = embed_kernel_name(args.copy, w.K, bool(info["suffix_index"]))
    kname = kname_full.split()[0]
    traffic, traffic_note = profiled_traffic(
        w.name, kname, PIPE_SOURCES if kname in ("embed_pipe_kernel", "embed_walk_kernel")
        else EMBED_SOURCES, with_note=True)
    res = {
        "metric": METRIC,
        "value": world * n_tok / (ms_step * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded Zipf token streams and f-gram sets, N(0,0.02)-like bf16 rows)",
        "config": {
            **prefill_config(w, world),
            "l2": f"flushed between timed steps ({FLUSH_BYTES >> 20} MB write + read back); "
                  f"steps rotate over {N_BATCHES} batches",
            "timing": "CUDA events around each step's launch on its stream",
            "copy": args.copy,
        },
        "roofline": {
            "bound": "hbm",
            "achieved": achieved,
            "peak": hbm,
            "unit": "GB/s",
            "frac": achieved / hbm,
            "traffic": traffic,
            "traffic_note": traffic_note,
            "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)",
            "algorithmic_bytes_per_launch": bytes_launch,
            "kernel": kname_full,
        },
        "e2e": {
            "value": world * n_tok / (e2e_ms[False] * 1e-3),
            "unit": "tokens/s",
            "h2d_bytes_per_step": 4 * n_tok,
            "d2h_bytes_per_step": 4,
            "what": "pinned host tokens read by the scone_embed kernel over the host link, "
                    "scone_status (sync + status word read); embeddings end on the device "
                    "as in Sec. 4.3",
            "staged": {"value": world * n_tok / (e2e_ms[True] * 1e-3), "unit": "tokens/s",
                       "what": "the same with a cudaMemcpyAsync of the tokens to the device "
                               "before scone_embed"},
        },
        "gpu_launches": args.steps,
        "clocks": clocks.summary(),
        "wall_s_timed_region": wall,
        "kernel_ms_min": min(per_step_ms),
        "kernel_ms_median": statistics.median(per_step_ms),
        "match_len_hist": {str(i): int(c) for i, c in enumerate(hist)},
        "avg_match_len": float((hist * np.arange(len(hist))).sum() / max(1, hist.sum())),
        "table": {k: info[k] for k in ("n_slots", "slot_bytes", "table_bytes",
                                       "max_insert_probe", "F_bytes", "T_bytes", "n_markers",
                                       "suffix_index")},
        "setup_s": setup_s,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_baseline(w, fg_tok, fg_len, batches_np[0], F, T)
    table.close()
    return res


def embed_kernel_name(copy: str, K: int, suffix_index: bool = False) -> str:
    """The kernel scone_embed launches for a copy mode (16-byte slots, aligned rows)."""
    if copy == "bulk":
        return "embed_bulk_kernel (fused match + TMA bulk gather)"
    if copy == "split":
        return "embed_split_kernel (match warps feed copy warps through shared memory)"
    pipe = copy == "pipelined" or (copy == "auto" and K <= 5 and (K > 3 or suffix_index))
    if pipe and suffix_index:
        return ("embed_walk_kernel (the lengths walked one bucket at a time over the suffix "
                "index, interleaved into the copy)")
    if pipe:
        return "embed_pipe_kernel (next tile's match interleaved into the copy)"
    return "embed_kernel (fused match + gather)"


def prefill_config(w, world: int) -> dict:
    """The workload part of a prefill line's config (shared by both arms)."""
    return {
        "workload": (f"{w.name}: {w.B}x{w.L} tokens, {w.n_fgrams} f-grams "
                     f"(n=2..{w.K}), K={w.K}, d={w.d}, vocab {w.vocab}, "
                     f"Zipf({w.zipf_s}), F in HBM, load factor {w.load_factor}"),
        "global_batch_tokens": world * w.B * w.L,
        "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
    }


def host_F_for(o, batches, w, F_dev=None):
    """A host array [n_fgrams, d] holding the F rows that the oracle selects
    on these batches (untimed set-up of the CPU legs). It spans every row, but
    only the pages of the selected rows are ever written, so a 41 GB F
    commits a few GB at most. The rows come from the device copy when one is
    given, else from the host-side generator."""
    sel = np.unique(np.concatenate([o.select(b)[0].reshape(-1) for b in batches]))
    sel = sel[sel >= 0]
    Fh = np.zeros((max(w.n_fgrams, 1), w.d), np.uint16)     # lazily committed pages
    if sel.size == 0:
        return Fh
    if F_dev is not None:
        import torch

        for a in range(0, sel.size, 1 << 16):
            part = sel[a:a + (1 << 16)]
            idx = torch.from_numpy(part).to(F_dev.device)
            Fh[part] = F_dev.index_select(0, idx).cpu().numpy().view(np.uint16)
        return Fh
    import concurrent.futures as cf

    import synth

    chunks = np.array_split(sel, max(1, min(16, os.cpu_count() or 1) * 4))

    def fill(part):
        if part.size:
            Fh[part] = synth.rows_cpu(synth.F_seed(w), w.d, part)

    with cf.ThreadPoolExecutor(min(16, os.cpu_count() or 1)) as ex:
        list(ex.map(fill, chunks))
    return Fh


def cpu_baseline(w, fg_tok, fg_len, tok, F, T, budget_s: float = 10.0):
    """The oracle as it stands (single thread, std::map) on a bounded sample:
    whole passes over one batch until budget_s of CPU work is done. Beside it,
    the same oracle with the sequences split over one std::thread per core of
    this process's affinity set."""
    import oracle

    o = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab)
    Fh = host_F_for(o, [tok], w, F_dev=F)
    Th = T.cpu().numpy().view(np.uint16)

    def timed(seqs, threads, budget):
        toks, passes, t0 = 0, 0, time.perf_counter()
        while True:
            b = (passes * seqs) % tok.shape[0]
            sample = tok[b:b + seqs]
            o.embed(sample, Fh, Th, threads=threads)
            toks += sample.size
            passes += 1
            if time.perf_counter() - t0 >= budget:
                break
        return toks, passes, time.perf_counter() - t0

    seqs = max(1, min(tok.shape[0], int(4096 // w.L) or 1))
    toks, passes, dt = timed(seqs, 1, budget_s)
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    mseqs = tok.shape[0]                      # the whole batch per pass: work for every thread
    cores = max(1, min(cores or 1, mseqs))    # threads actually used
    mtoks, mpasses, mdt = timed(mseqs, cores, budget_s / 2)
    return {"value": toks / dt, "unit": "tokens/s", "cores": 1, "kind": "oracle",
            "sample": f"{passes} oracle passes of {seqs} x {w.L} tokens of the same workload "
                      f"({toks} tokens, {dt:.1f} s, map build untimed)",
            "threads": {"value": mtoks / mdt, "unit": "tokens/s", "cores": cores,
                        "kind": "oracle, sequences split over std::threads",
                        "sample": f"{mpasses} passes of {mseqs} x {w.L} tokens "
                                  f"({mtoks} tokens, {mdt:.1f} s)"}}


# ------------------------------------------------------- offloaded decode
def host_link_bandwidth(dev, table, F_rows: int, d: int, zero_copy: bool = True):
    """Host -> device bandwidth, measured two ways; the larger is the roofline.

    copy: pinned cudaMemcpyAsync of 1 GiB, best of 10.
    zero_copy: the library's gather kernel streaming consecutive rows of the
    host-mapped F (device loads over the host link), 1 GiB, best of 10.
    zero_copy_random (reported, not the roofline): the same kernel reading
    1 GiB of rows drawn uniformly from all of F.
    """
    import torch

    import paper_2502_01637_gb300 as scone

    nb = 1 << 30
    src = torch.empty(nb, dtype=torch.uint8).pin_memory()
    dst = torch.empty(nb, dtype=torch.uint8, device=dev)
    best_copy = best_d2h = 0.0
    for _ in range(10):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        dst.copy_(src, non_blocking=True)
        b.record()
        b.synchronize()
        best_copy = max(best_copy, nb / (a.elapsed_time(b) * 1e-3) / 1e9)
    for _ in range(10):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        src.copy_(dst, non_blocking=True)
        b.record()
        b.synchronize()
        best_d2h = max(best_d2h, nb / (a.elapsed_time(b) * 1e-3) / 1e9)
    del dst
    if not zero_copy:
        return {"copy_gbs": best_copy, "d2h_copy_gbs": best_d2h, "peak_gbs": best_copy}
    n = min(F_rows, nb // (2 * d))
    tok = torch.zeros(n, dtype=torch.int32, device=dev)
    out = torch.empty((n, d), dtype=torch.int16, device=dev)

    def gather_rate(row):
        best = 0.0
        for _ in range(10):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            scone.scone_embed_gather(table, tok, row, out)
            b.record()
            b.synchronize()
            best = max(best, n * 2 * d / (a.elapsed_time(b) * 1e-3) / 1e9)
        return best

    best_zc = gather_rate(torch.arange(n, dtype=torch.int32, device=dev))
    rnd = np.random.default_rng(1).integers(0, F_rows, n).astype(np.int32)
    best_rand = gather_rate(torch.from_numpy(rnd).to(dev))
    scone.scone_status(table)
    return {"copy_gbs": best_copy, "zero_copy_gbs": best_zc,
            "zero_copy_random_gbs": best_rand, "peak_gbs": max(best_copy, best_zc),
            "d2h_copy_gbs": best_d2h}


def decode_row_ceiling(table, new_d, rows, host_bytes, d):
    """What the host link gives for the rows the decode steps select, without
    the steps' dependent match: every step's rows gathered in one launch
    (best of 5), and gathered one step per launch in a CUDA graph (best of 5
    replays; the per-step time left to the match is the decode step's time
    minus this one)."""
    import torch

    import paper_2502_01637_gb300 as scone

    steps, S = rows.shape
    big = torch.empty((steps * S, d), dtype=torch.int16, device=new_d.device)
    one = torch.empty((S, d), dtype=torch.int16, device=new_d.device)
    flat_tok, flat_row = new_d.reshape(-1).contiguous(), rows.reshape(-1).contiguous()

    def best(fn, n=5):
        t = []
        for _ in range(n):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            b.synchronize()
            t.append(a.elapsed_time(b))
        return min(t)

    scone.scone_embed_gather(table, flat_tok, flat_row, big)
    all_ms = best(lambda: scone.scone_embed_gather(table, flat_tok, flat_row, big))
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for k in range(steps):
            scone.scone_embed_gather(table, new_d[k], rows[k], one)
    g.replay()
    step_ms = best(g.replay) / steps
    scone.scone_status(table)
    del big, g
    return {"all_steps_one_launch_gbs": host_bytes / (all_ms * 1e-3) / 1e9,
            "per_step_gather_us": step_ms * 1e3,
            "per_step_gather_gbs": host_bytes / steps / (step_ms * 1e-3) / 1e9,
            "what": "the host rows the decode selects, gathered by gather_kernel without "
                    "the match: all steps in one launch, and one launch per step (graph)"}


def bench_decode(args, world, rank, local):
    import torch

    import synth
    import paper_2502_01637_gb300 as scone

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = workload(args.workload)
    t0 = time.time()
    fg_tok, fg_len, _ = synth.fgram_set(w)
    stream = torch.cuda.current_stream()
    buf = scone.scone_host_alloc(w.n_fgrams * w.d * 2)
    synth.rows_gpu(synth.F_seed(w), w.d, 0, w.n_fgrams, buf.ptr, stream.cuda_stream)
    T = torch.empty((w.vocab, w.d), dtype=torch.int16, device=dev)
    synth.rows_gpu(synth.T_seed(w), w.d, 0, w.vocab, T.data_ptr(), stream.cuda_stream)
    table = scone.scone_table_build(fg_tok, fg_len, w.K, w.vocab, w.d, buf.ptr, T,
                                    F_location=scone.SCONE_ROWS_HOST_MAPPED)
    setup_s = time.time() - t0
    link = host_link_bandwidth(dev, table, w.n_fgrams, w.d)
    # decode steps move rows with register loads (AUTO) or TMA bulk copies (--copy bulk)
    scone.scone_table_set_copy_mode(table, scone.SCONE_COPY_BULK if args.copy == "bulk"
                                    else scone.SCONE_COPY_AUTO)
    hist, hl, new = synth.decode_inputs(w)
    S, steps = w.dec_S, w.dec_steps
    new_d = torch.from_numpy(new).to(dev)
    out = torch.empty((S, w.d), dtype=torch.int16, device=dev)
    lens = torch.empty((steps, S), dtype=torch.uint8, device=dev)
    rows = torch.empty((steps, S), dtype=torch.int32, device=dev)
    # one eager pass: match lengths of every step (host bytes = matched rows)
    st = scone.scone_decode_create(table, hist, hl)
    for k in range(steps):
        scone.scone_decode_step(st, new_d[k], out, rows[k], lens[k])
    scone.scone_status(table)
    ln = lens.cpu().numpy()
    matched = int((ln >= 2).sum())
    hist_counts = np.bincount(ln.reshape(-1), minlength=w.K + 1)
    st.close()
    step_rows = decode_row_ceiling(table, new_d, rows, matched * 2 * w.d, w.d)
    # timed: the 256-step loop captured once in a CUDA graph, replayed
    st = scone.scone_decode_create(table, hist, hl)
    for k in range(3):
        scone.scone_decode_step(st, new_d[k], out)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for k in range(steps):
            scone.scone_decode_step(st, new_d[k], out)
    replays = max(10, args.steps // steps)
    for _ in range(max(1, args.warmup // steps) + 1):
        g.replay()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(replays)]
    clocks = ClockSampler(local)
    torch.cuda.synchronize()
    with clocks:
        for r in range(replays):
            ev[r][0].record()
            g.replay()
            ev[r][1].record()
        torch.cuda.synchronize()
    scone.scone_status(table)
    per_replay = [a.elapsed_time(b) for a, b in ev]
    ms_step = statistics.mean(per_replay) / steps

    # end to end through the public API, one step at a time: the step's new
    # tokens from pinned host memory (read by the kernel; "staged": copied to
    # the device first), scone_decode_step, scone_status (sync + status word)
    host_new = torch.from_numpy(new).pin_memory()
    tok_d = torch.empty(S, dtype=torch.int32, device=dev)
    e2e_n = min(steps, 64)
    e2e_ms = {}
    raw_stream = torch.cuda.current_stream().cuda_stream
    for staged in (False, True):
        e2e_t = []
        for k in range(e2e_n + 3):
            torch.cuda.synchronize()
            t1 = time.perf_counter()
            if staged:
                tok_d.copy_(host_new[k % steps], non_blocking=True)
                scone.scone_decode_step(st, tok_d, out, stream=raw_stream)
            else:
                scone.scone_decode_step(st, host_new[k % steps], out, stream=raw_stream)
            scone.scone_status(table, raw_stream)
            if k >= 3:
                e2e_t.append(time.perf_counter() - t1)
        e2e_ms[staged] = max_over_ranks(1e3 * statistics.mean(e2e_t), world)
    host_bytes_step = matched / steps * 2 * w.d
    hbm_bytes_step = (S * (4 + 32 * (w.K - 1)) + (S - matched / steps) * 2 * w.d + S * 2 * w.d)
    achieved = host_bytes_step / (ms_step * 1e-3) / 1e9
    fracs = [host_bytes_step * steps / (t * 1e-3) / 1e9 / link["peak_gbs"] for t in per_replay]
    res = {
        "metric": METRIC,
        "value": S / (ms_step * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": replays * steps,
        "warmup": args.warmup,
        "ms_per_step": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded Zipf histories, tokens and f-gram set)",
        "config": {
            "workload": (f"{w.name}: {S} live sequences x {steps} decode steps, "
                         f"{w.n_fgrams} f-grams (n=2..{w.K}), d={w.d}, vocab {w.vocab}, "
                         f"F ({w.n_fgrams * w.d * 2 / 1e9:.1f} GB) host-pinned, device-mapped, "
                         f"rows in {w.row_order.replace('_', '-')} order"),
            "timing": f"{steps} steps captured in one CUDA graph, {replays} replays, "
                      "CUDA events per replay",
            "l2": "working set per replay (~%d MB of rows) exceeds L2" %
                  (steps * S * 2 * w.d * 2 >> 20),
        },
        "roofline": {
            "bound": "host-link",
            "achieved": achieved,
            "peak": link["peak_gbs"],
            "unit": "GB/s",
            "frac": achieved / link["peak_gbs"],
            "traffic": None,
            "peak_source": "measured in this run: max(pinned 1 GiB H2D copy, zero-copy "
                           "streaming read by the gather kernel)",
            "host_link": link,
            "decode_rows": step_rows,
            "host_bytes_per_step": host_bytes_step,
            "hbm_bytes_per_step": hbm_bytes_step,
            "kernel": ("decode_kernel (one warp per sequence, TMA bulk row copies)"
                       if args.copy == "bulk" else "decode_kernel (one warp per sequence)"),
        },
        "e2e": {"value": world * S / (e2e_ms[False] * 1e-3), "unit": "tokens/s",
                "h2d_bytes_per_step": 4 * S, "d2h_bytes_per_step": 4,
                "what": "each step: new tokens read by the decode kernel from pinned host "
                        "memory, scone_decode_step, scone_status (sync + status word read); "
                        "no graph, one step at a time as a serving loop issues them",
                "staged": {"value": world * S / (e2e_ms[True] * 1e-3), "unit": "tokens/s",
                           "what": "the same with a cudaMemcpyAsync of the tokens first"}},
        "gpu_launches": replays * steps,
        "clocks": clocks.summary(),
        "match_len_hist": {str(i): int(c) for i, c in enumerate(hist_counts)},
        "match_rate": matched / (S * steps),
        "replay_frac": {"median": statistics.median(fracs), "min": min(fracs),
                        "max": max(fracs), "replays": replays,
                        "what": "host-link fraction of each graph replay (256 steps)"},
        "setup_s": setup_s,
    }
    st.close()
    table.close()
    buf.free()
    return res


# --------------------------------------------------- training-time pre-scan
def bench_prescan(args, world, rank, local):
    """scone_match over a corpus in host memory: tokens read and (row, len)
    tags written through host-mapped addresses by the match kernel."""
    import torch

    import synth
    import paper_2502_01637_gb300 as scone

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = workload(args.workload)
    n = w.B * w.L
    t0 = time.time()
    fg_tok, fg_len, _ = synth.fgram_set(w)
    F = torch.zeros((w.n_fgrams, w.d), dtype=torch.int16, device=dev)
    T = torch.zeros((w.vocab, w.d), dtype=torch.int16, device=dev)
    table = scone.scone_table_build(fg_tok, fg_len, w.K, w.vocab, w.d, F, T,
                                    load_factor=w.load_factor)
    corpus = scone.scone_host_alloc(n * 4)
    tags_len = scone.scone_host_alloc(n)
    tags_row = scone.scone_host_alloc(n * 4)
    synth.query_tokens(w, out=corpus.numpy(np.int32)[:n].reshape(w.B, w.L))
    setup_s = time.time() - t0
    link = host_link_bandwidth(dev, table, w.n_fgrams, w.d, zero_copy=False)
    lib = scone.load_library()
    stream = torch.cuda.current_stream()

    def staged():
        # chunks of whole sequences copied in, tagged in HBM, tags copied out
        rc = lib.scone_prescan(table.handle, corpus.ptr, w.B, w.L, tags_row.ptr, tags_len.ptr, 0,
                               stream.cuda_stream)
        assert rc == 0

    def zero_copy():
        # the match kernel reading the tokens and writing the tags in host memory
        rc = lib.scone_match(table.handle, corpus.ptr, w.B, w.L, tags_row.ptr, tags_len.ptr,
                             stream.cuda_stream)
        assert rc == 0

    def timed(step, clocks=None):
        for _ in range(args.warmup):
            step()
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(args.steps)]
        if clocks is not None:
            clocks.__enter__()
        for k in range(args.steps):
            ev[k][0].record(stream)
            step()
            ev[k][1].record(stream)
        torch.cuda.synchronize()
        if clocks is not None:
            clocks.__exit__(None, None, None)
        return statistics.mean(a.elapsed_time(b) for a, b in ev)

    zc_ms = timed(zero_copy)
    clocks = ClockSampler(local)
    ms = timed(staged, clocks)
    scone.scone_status(table)
    h2d = 4 * n / (ms * 1e-3) / 1e9
    d2h = 5 * n / (ms * 1e-3) / 1e9
    lens = np.bincount(tags_len.numpy(np.uint8)[:n], minlength=w.K + 1)
    res = {
        "metric": METRIC,
        "value": n / (ms * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "int32",
        "data": "synthetic corpus (seeded Zipf sequences) and f-gram set",
        "config": {"workload": (f"{w.name}: pre-scan of {w.B} x {w.L} = {n} corpus tokens in "
                                f"host memory, {w.n_fgrams} f-grams (n=2..{w.K}); tags row "
                                "(int32) and len (uint8) written to host memory"),
                   "timing": "CUDA events on the caller's stream around each full-corpus "
                             "scone_prescan (chunks of 32 Mi tokens staged through HBM)"},
        "roofline": {
            "bound": "host-link",
            "achieved": h2d,
            "peak": link["copy_gbs"],
            "unit": "GB/s",
            "frac": max(h2d / link["copy_gbs"], d2h / link["d2h_copy_gbs"]),
            "traffic": None,
            "d2h_achieved": d2h,
            "host_link": link,
            "kernel": ("match_walk_kernel on HBM chunks, with the copies in and out "
                       "(scone_prescan)"),
        },
        "zero_copy": {"value": n / (zc_ms * 1e-3), "unit": "tokens/s", "ms_per_step": zc_ms,
                      "what": "scone_match on the host addresses (match_kernel reading tokens "
                              "and writing tags over the host link)"},
        "gpu_launches": args.steps * -(-n // ((32 << 20) // w.L * w.L)),
        "clocks": clocks.summary(),
        "match_len_hist": {str(i): int(c) for i, c in enumerate(lens)},
        "setup_s": setup_s,
    }
    table.close()
    corpus.free()
    tags_len.free()
    tags_row.free()
    return res


# ------------------------------------------------ decode with F in a file
def bench_store(args, world, rank, local):
    """Decode steps with F in a file (the storage tier): 512 live sequences,
    each step selects on the GPU (scone_decode_step without rows), then
    scone_rowstore_gather copies cached rows and reads the missed ones from
    the file (O_DIRECT, 4 KiB rows) into the HBM cache. 2e6 f-grams, d = 2048
    (an 8.2 GB file); cache of 65,536 rows (256 MiB of HBM)."""
    import torch

    import synth
    import paper_2502_01637_gb300 as scone

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = workload("decode_profile")
    cache_rows = 65536
    t0 = time.time()
    fg_tok, fg_len, _ = synth.fgram_set(w)
    path = os.path.join(ROOT, "_store_F.bin")
    rows_per = 1 << 16
    with open(path, "wb") as f:
        for r0 in range(0, w.n_fgrams, rows_per):
            synth.rows_range_cpu(synth.F_seed(w), w.d, r0,
                                 min(rows_per, w.n_fgrams - r0)).tofile(f)
    os.sync()
    stream = torch.cuda.current_stream()
    T = torch.empty((w.vocab, w.d), dtype=torch.int16, device=dev)
    synth.rows_gpu(synth.T_seed(w), w.d, 0, w.vocab, T.data_ptr(), stream.cuda_stream)
    F_stub = torch.zeros((1, w.d), dtype=torch.int16, device=dev)
    table = scone.scone_table_build(fg_tok, fg_len, w.K, w.vocab, w.d, F_stub, T)
    store = scone.RowStore(path, w.n_fgrams, w.d, cache_rows)
    setup_s = time.time() - t0
    hist, hl, new = synth.decode_inputs(w)
    S, steps = w.dec_S, w.dec_steps
    new_d = torch.from_numpy(new).to(dev)
    out = torch.empty((S, w.d), dtype=torch.int16, device=dev)
    row = torch.empty(S, dtype=torch.int32, device=dev)
    lib = scone.load_library()
    st = scone.scone_decode_create(table, hist, hl)

    def step(k):
        rc = lib.scone_decode_step(st.handle, new_d[k % steps].data_ptr(), None, row.data_ptr(),
                                   None, stream.cuda_stream)
        assert rc == 0
        scone.scone_rowstore_gather(store, table, new_d[k % steps], row, out)

    for k in range(args.warmup):
        step(k)
    s0 = store.stats()
    n_steps = max(args.steps, 1)
    clocks = ClockSampler(local)
    torch.cuda.synchronize()
    with clocks:
        t1 = time.perf_counter()
        for k in range(n_steps):
            step(args.warmup + k)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t1
    scone.scone_status(table)
    s1 = store.stats()
    ms = 1e3 * wall / n_steps
    # the file's own random-row rate with the store's threads and I/O mode
    probe = scone.scone_rowstore_probe_reads(store, 100_000, seed=7)
    misses = s1["misses"] - s0["misses"]
    positions = s1["positions"] - s0["positions"]
    rows_read = s1["rows_read"] - s0["rows_read"]
    res = {
        "metric": "embedded tokens/s at 1 GB300, F in a file (storage tier), decode",
        "value": world * S / (ms * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": n_steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded Zipf decode tokens; F rows written to a file on the box)",
        "config": {"workload": (f"store_decode: {S} sequences per step, {w.n_fgrams} f-grams, "
                                f"d={w.d}, F in an {w.n_fgrams * w.d * 2 / 1e9:.1f} GB file, "
                                f"HBM row cache of {cache_rows} rows"),
                   "timing": "host wall clock per step (each step synchronizes: the host "
                             "reads the misses)",
                   "io": "O_DIRECT pread" if s1["direct_io"] else "buffered pread"},
        "roofline": {"bound": "storage", "achieved": rows_read * w.d * 2 / wall / 1e9,
                     "peak": probe["bytes_per_s"] / 1e9, "unit": "GB/s read from the file",
                     "frac": rows_read * w.d * 2 / wall / probe["bytes_per_s"],
                     "traffic": None,
                     "peak_source": ("measured in this run: 100,000 uniformly drawn rows of "
                                     "the same file read by the store's reader threads with "
                                     "its I/O mode (scone_rowstore_probe_reads)"),
                     "probe_rows_per_s": probe["rows_per_s"],
                     "step_rows_per_s": rows_read / wall,
                     "kernel": "lookup_kernel + file reads + fill_kernel (host-driven)"},
        "store": {"hit_rate": 1.0 - misses / max(1, positions), "positions": positions,
                  "misses": misses, "rows_read": rows_read,
                  "rows_read_per_step": rows_read / n_steps,
                  "direct_io": bool(s1["direct_io"])},
        "e2e": {"value": world * S / (ms * 1e-3), "unit": "tokens/s",
                "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0,
                "what": "decode tokens already on the device; the timed loop includes the "
                        "host's file reads"},
        "gpu_launches": n_steps * 3,
        "clocks": clocks.summary(),
        "setup_s": setup_s,
    }
    st.close()
    store.close()
    table.close()
    os.remove(path)
    return res


# ------------------------------------------------------ mixed serving batch
def mixed_batch(w, k, n_prefill_seq=48, n_decode=512):
    """Batch k of a serving step over the prefill_1b law: n_prefill_seq prompt
    chunks of seeded ragged lengths and n_decode one-token decode chunks, the
    same 65,536 tokens as a prefill_1b batch. Returns (tokens, cu_seqlens,
    slot of each sequence)."""
    import synth

    n_tok = w.B * w.L
    rng = np.random.default_rng(1000 + k)
    raw = rng.uniform(0.25, 1.75, n_prefill_seq)
    lens = np.floor(raw / raw.sum() * (n_tok - n_decode)).astype(np.int64)
    lens[0] += n_tok - n_decode - lens.sum()
    lens = np.concatenate([lens, np.ones(n_decode, np.int64)])
    order = rng.permutation(lens.size)               # prefill and decode chunks interleaved
    lens = lens[order]
    tok = synth.query_tokens(w.scaled(w.name + "_mixed", B=1, L=n_tok), range(k, k + 1))[0]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    slots = rng.permutation(2048)[:lens.size].astype(np.int32)
    return tok, cu, slots


def bench_mixed(args, world, rank, local):
    """scone_embed_varlen on mixed serving batches: chunked-prefill pieces and
    decode tokens of 560 sequences in one launch, continuing 2048 slots of a
    decode state (the prefill_1b table, F and T)."""
    import torch

    import synth
    import paper_2502_01637_gb300 as scone

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = synth.WORKLOADS["prefill_1b"]
    n_tok = w.B * w.L
    t0 = time.time()
    fg_tok, fg_len, _ = synth.fgram_set(w)
    stream = torch.cuda.current_stream()
    F = torch.empty((w.n_fgrams, w.d), dtype=torch.int16, device=dev)
    T = torch.empty((w.vocab, w.d), dtype=torch.int16, device=dev)
    synth.rows_gpu(synth.F_seed(w), w.d, 0, w.n_fgrams, F.data_ptr(), stream.cuda_stream)
    synth.rows_gpu(synth.T_seed(w), w.d, 0, w.vocab, T.data_ptr(), stream.cuda_stream)
    table = scone.scone_table_build(fg_tok, fg_len, w.K, w.vocab, w.d, F, T,
                                    load_factor=w.load_factor)
    S = 2048
    H = w.K - 1
    hist0 = synth.query_tokens(w.scaled("mixed_hist", B=S, L=H))
    state = scone.scone_decode_create(table, hist0, np.full(S, H, np.int32))
    batches = [mixed_batch(w, k) for k in range(N_BATCHES)]
    dev_b = [(torch.from_numpy(t).to(dev), torch.from_numpy(c).to(dev), torch.from_numpy(s).to(dev))
             for t, c, s in batches]
    out = torch.empty((n_tok, w.d), dtype=torch.int16, device=dev)
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    setup_s = time.time() - t0

    def step(k):
        t, c, s_ = dev_b[k % N_BATCHES]
        scone.scone_embed_varlen(table, t, c, out, state=state, seq_slot=s_)

    for k in range(args.warmup):
        flush_l2(flush)
        step(k)
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    clocks = ClockSampler(local)
    barrier(world)
    with clocks:
        for k in range(args.steps):
            flush_l2(flush)
            ev[k][0].record(stream)
            step(k)
            ev[k][1].record(stream)
        torch.cuda.synchronize()
    barrier(world)
    scone.scone_status(table)
    per_step_ms = [a.elapsed_time(b) for a, b in ev]
    kernel_ms = statistics.mean(per_step_ms)
    ms_step = max_over_ranks(kernel_ms, world)

    # end to end: pinned tokens, offsets and slots in; status word out
    host_b = [tuple(torch.from_numpy(x).pin_memory() for x in b) for b in batches]
    e2e_t = []
    for k in range(max(3, min(args.steps, 50))):
        flush_l2(flush)
        torch.cuda.synchronize()
        t1 = time.perf_counter()
        t, c, s_ = dev_b[0]
        for d_, h_ in zip((t, c, s_), host_b[k % N_BATCHES]):
            d_[:h_.numel()].copy_(h_, non_blocking=True)
        scone.scone_embed_varlen(table, t, c, out, state=state, seq_slot=s_)
        scone.scone_status(table)
        e2e_t.append(time.perf_counter() - t1)
    e2e_ms = max_over_ranks(1e3 * statistics.mean(e2e_t), world)
    n_seq = batches[0][1].size - 1
    per_tok = algorithmic_bytes_per_token(w.K, w.d)
    bytes_launch = per_tok * n_tok
    hbm, peak_src = measured_peaks()
    achieved = bytes_launch / (kernel_ms * 1e-3) / 1e9
    res = {
        "metric": METRIC,
        "value": world * n_tok / (ms_step * 1e-3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded Zipf token streams and f-gram sets, N(0,0.02)-like bf16 rows)",
        "config": {
            "workload": (f"mixed_serving: {n_tok} tokens per launch in {n_seq} sequences "
                         f"(48 ragged prompt chunks + 512 one-token decode chunks), each "
                         f"continuing one of {S} decode-state slots; prefill_1b table "
                         f"({w.n_fgrams} f-grams, K={w.K}, d={w.d}), F in HBM"),
            "l2": f"flushed between timed steps ({FLUSH_BYTES >> 20} MB write + read back); "
                  f"steps rotate over {N_BATCHES} batches",
            "timing": "CUDA events around each step (embedding and history launches)",
        },
        "roofline": {
            "bound": "hbm",
            "achieved": achieved,
            "peak": hbm,
            "unit": "GB/s",
            "frac": achieved / hbm,
            "traffic": (profiled_traffic("mixed_serving", "varlen_walk_kernel", VARLEN_SOURCES)
                        if table.info()["suffix_index"] else None),
            "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)",
            "algorithmic_bytes_per_launch": bytes_launch,
            "kernel": ("varlen_walk_kernel (fused match + gather over packed sequences, the "
                       "lengths walked over the suffix index)" if table.info()["suffix_index"]
                       else "varlen_embed_kernel (fused match + gather over packed sequences)"),
        },
        "e2e": {
            "value": world * n_tok / (e2e_ms * 1e-3),
            "unit": "tokens/s",
            "h2d_bytes_per_step": 4 * n_tok + 4 * (n_seq + 1) + 4 * n_seq,
            "d2h_bytes_per_step": 4,
            "what": "pinned tokens, offsets and slots -> device, scone_embed_varlen, "
                    "scone_status",
        },
        "gpu_launches": args.steps,   # one varlen kernel per step (it also rewrites the histories)
        "clocks": clocks.summary(),
        "kernel_ms_min": min(per_step_ms),
        "setup_s": setup_s,
    }
    state.close()
    table.close()
    return res


# ------------------------------------------------------- F precompute (NEXT-3)
def model_flops_per_token(m) -> int:
    """Dense-layer FLOPs of one token through the f-gram model (2 per MAC)."""
    return 2 * m.n_layers * (4 * m.d * m.d + 3 * m.d * m.ffw)


def bench_precompute(args, world, rank, local):
    """F rows of 65,536 f-grams (prefill_1b's list: 2- and 3-grams) by the
    12-layer, d = 2048 f-gram model (the paper's 711M OLMo shape, random
    weights): one step is one scone_fgram_precompute call."""
    import torch

    import synth
    import paper_2502_01637_gb300 as scone

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = synth.WORKLOADS["prefill_1b"]
    m = synth.MODELS["olmo_711m"]
    n_f = 65536
    t0 = time.time()
    fg_tok, fg_len, _ = synth.fgram_set(w)
    fg_tok, fg_len = fg_tok[:n_f], fg_len[:n_f]
    stream = torch.cuda.current_stream()
    weights = torch.empty(m.n_elems, dtype=torch.int16, device=dev)
    synth.model_weights_gpu(m, weights.data_ptr(), stream.cuda_stream)
    T = torch.empty((w.vocab, m.d), dtype=torch.int16, device=dev)
    synth.rows_gpu(synth.T_seed(w), m.d, 0, w.vocab, T.data_ptr(), stream.cuda_stream)
    tok_d = torch.from_numpy(fg_tok).to(dev)
    len_d = torch.from_numpy(fg_len).to(dev)
    F = torch.empty((n_f, m.d), dtype=torch.int16, device=dev)
    model = scone.FgramModel(m.d, m.n_heads, m.ffw, m.n_layers, weights, batch=16384,
                             max_pos=m.max_pos)
    setup_s = time.time() - t0
    tokens = int(fg_len.astype(np.int64).sum())
    flops = model_flops_per_token(m) * tokens

    def step():
        scone.scone_fgram_precompute(model, tok_d, len_d, T, F)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    clocks = ClockSampler(local)
    barrier(world)
    with clocks:
        for k in range(args.steps):
            ev[k][0].record(stream)
            step()
            ev[k][1].record(stream)
        torch.cuda.synchronize()
    barrier(world)
    ms = max_over_ranks(statistics.mean(a.elapsed_time(b) for a, b in ev), world)

    # the dominant kernel timed alone with CUDA events: the gate/up GEMM of one
    # 16,384-f-gram batch (M = its tokens, N = 2 ffw, K = d) with SwiGLU
    M = int(fg_len[:16384].astype(np.int64).sum())
    A = torch.empty((M, m.d), dtype=torch.int16, device=dev)
    synth.rows_gpu(99, m.d, 0, M, A.data_ptr(), stream.cuda_stream)
    Bw = weights[m.offset(0, "gu"):m.offset(0, "gu") + 2 * m.ffw * m.d].view(2 * m.ffw, m.d)
    C = torch.empty((M, m.ffw), dtype=torch.int16, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    for _ in range(3):
        scone.scone_gemm_bf16(A, Bw, C, epilogue=scone.SCONE_GEMM_SWIGLU, status=status)
    gev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(20)]
    for a, b in gev:
        a.record(stream)
        scone.scone_gemm_bf16(A, Bw, C, epilogue=scone.SCONE_GEMM_SWIGLU, status=status)
        b.record(stream)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    g_ms = statistics.mean(a.elapsed_time(b) for a, b in gev)
    g_tflops = 2.0 * M * 2 * m.ffw * m.d / (g_ms * 1e-3) / 1e12
    peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json"))) \
        if os.path.exists(os.path.join(ROOT, "MEASURED_PEAKS.json")) else {}
    peak = float(peaks.get("bf16_tflops", 1900.0))
    res = {
        "metric": "precomputed F rows/s at 1 GB300 (f-gram model forward, Sec. 3.2)",
        "value": world * n_f / (ms * 1e-3),
        "unit": "f-gram rows/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (random bf16 weights, seeded f-gram list and T rows)",
        "config": {"workload": (f"precompute: {n_f} f-grams ({tokens} tokens) of prefill_1b's "
                                f"list through a {m.n_layers}-layer model, d={m.d}, "
                                f"{m.n_heads} heads, ffw={m.ffw} (SwiGLU), "
                                f"{m.n_elems / 1e6:.0f}M parameters; batches of 16384 f-grams"),
                   "l2": "weights (1.6 GB) and activations far larger than L2; no flush",
                   "timing": "CUDA events around each scone_fgram_precompute call"},
        "model_tflops": flops / (ms * 1e-3) / 1e12,
        "roofline": {
            "bound": "tensor",
            "achieved": g_tflops,
            "peak": peak,
            "unit": "TFLOP/s",
            "frac": g_tflops / peak,
            "traffic": None,
            "peak_source": "measured (MEASURED_PEAKS.json bf16_tflops, burst)" if peaks
                           else "fallback",
            "kernel": f"gemm_bf16_kernel<SWIGLU>: M={M}, N={2 * m.ffw}, K={m.d} "
                      "(gate/up of one batch), timed alone",
            "kernel_ms": g_ms,
            "algorithmic_flops_per_launch": 2 * M * 2 * m.ffw * m.d,
        },
        "e2e": {"value": world * n_f / (ms * 1e-3), "unit": "f-gram rows/s",
                "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0,
                "what": "the f-gram list and F stay on the device (F is written where the "
                        "table will read it)"},
        "gpu_launches": args.steps * (4 * (3 + m.n_layers * 7)),
        "clocks": clocks.summary(),
        "setup_s": setup_s,
    }
    if rank == 0 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_baseline_precompute(m, fg_tok, fg_len, w)
    model.close()
    return res


def bench_gemm(args, world, rank, local):
    """The tensor-core GEMM alone at the f-gram model's gate/up shape with the
    SwiGLU epilogue (M = 16384 tokens, N = 2 ffw = 16384, K = d = 2048): the
    case the ncu summaries of the kernel are taken on."""
    import torch

    import synth
    import paper_2502_01637_gb300 as scone

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    M, N, K = 16384, 16384, 2048
    A = torch.empty((M, K), dtype=torch.int16, device=dev)
    B = torch.empty((N, K), dtype=torch.int16, device=dev)
    synth.rows_gpu(5, K, 0, M, A.data_ptr(), stream.cuda_stream)
    synth.rows_gpu(6, K, 0, N, B.data_ptr(), stream.cuda_stream)
    C = torch.empty((M, N // 2), dtype=torch.int16, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)

    def step():
        scone.scone_gemm_bf16(A, B, C, epilogue=scone.SCONE_GEMM_SWIGLU, status=status)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    clocks = ClockSampler(local)
    with clocks:
        for a, b in ev:
            a.record(stream)
            step()
            b.record(stream)
        torch.cuda.synchronize()
    assert int(status.item()) == 0
    ms = statistics.mean(a.elapsed_time(b) for a, b in ev)
    flops = 2.0 * M * N * K
    # the one-SM-per-tile kernel on the same operands, for comparison
    for _ in range(3):
        scone.scone_gemm_bf16(A, B, C, epilogue=scone.SCONE_GEMM_SWIGLU, status=status, variant=1)
    ev1 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(10)]
    for a, b in ev1:
        a.record(stream)
        scone.scone_gemm_bf16(A, B, C, epilogue=scone.SCONE_GEMM_SWIGLU, status=status, variant=1)
        b.record(stream)
    torch.cuda.synchronize()
    ms1 = statistics.mean(a.elapsed_time(b) for a, b in ev1)
    # context: cuBLAS (torch.matmul, bf16, plain store) on the same shape, and on
    # the 8192^3 shape the measured peak is quoted on
    def cublas_tflops(m, n, k, reps=10):
        a = torch.randn((m, k), dtype=torch.bfloat16, device=dev)
        b = torch.randn((n, k), dtype=torch.bfloat16, device=dev)
        for _ in range(3):
            torch.matmul(a, b.t())
        e = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
             for _ in range(reps)]
        for x, y in e:
            x.record(stream)
            torch.matmul(a, b.t())
            y.record(stream)
        torch.cuda.synchronize()
        best = min(x.elapsed_time(y) for x, y in e)
        return 2.0 * m * n * k / (best * 1e-3) / 1e12

    cublas_same = cublas_tflops(M, N, K)
    cublas_8192 = cublas_tflops(8192, 8192, 8192)
    peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json"))) \
        if os.path.exists(os.path.join(ROOT, "MEASURED_PEAKS.json")) else {}
    peak = float(peaks.get("bf16_tflops", 1900.0))
    tf = flops / (ms * 1e-3) / 1e12
    return {
        "metric": "bf16 GEMM TFLOP/s at 1 GB300 (tcgen05, SwiGLU epilogue)",
        "value": tf, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"gemm_profile: M={M}, N={N}, K={K}, C = silu(gate) up "
                               f"[{M} x {N // 2}]",
                   "l2": "operands 134 MB, output 268 MB (larger than L2); no flush"},
        "roofline": {"bound": "tensor", "achieved": tf, "peak": peak, "unit": "TFLOP/s",
                     "frac": tf / peak, "traffic": None,
                     "peak_source": "measured (MEASURED_PEAKS.json bf16_tflops, burst)"
                                    if peaks else "fallback",
                     "kernel": "gemm_bf16_kernel<SWIGLU>",
                     "algorithmic_flops_per_launch": flops},
        "e2e": {"value": tf, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0, "what": "operands stay on the device"},
        "gpu_launches": args.steps, "clocks": clocks.summary(),
        "variants": {"sm_pairs_256x256 (default)": tf,
                     "one_sm_128x256": flops / (ms1 * 1e-3) / 1e12},
        "cublas_context": {"same_shape_plain_store_tflops": cublas_same,
                           "shape_8192_cubed_tflops": cublas_8192,
                           "what": "torch.matmul bf16, best of 10, CUDA events; context for "
                                   "the roofline, whose peak stays MEASURED_PEAKS.json's"},
    }


def cpu_baseline_precompute(m, fg_tok, fg_len, w, budget_s: float = 10.0):
    """The float64 oracle forward (numpy; its BLAS may use several threads) on
    the first f-grams of the same list, until about budget_s."""
    import synth
    from oracle import fgram_model as fm

    packed = synth.model_weights_cpu(m)
    W = fm.Weights(packed, m)
    used = np.unique(fg_tok[:64][fg_tok[:64] >= 0])
    T = np.zeros((w.vocab, m.d), np.uint16)
    T[used] = synth.rows_cpu(synth.T_seed(w), m.d, used)
    t0 = time.perf_counter()
    done = 0
    while done < 64:
        fm.fgram_row(fg_tok[done][:fg_len[done]], T, W, emulate_bf16=True)
        done += 1
        if time.perf_counter() - t0 >= budget_s:
            break
    dt = time.perf_counter() - t0
    return {"value": done / dt, "unit": "f-gram rows/s", "cores": os.cpu_count() or 1,
            "kind": "oracle",
            "sample": f"float64 oracle forward of the first {done} f-grams ({dt:.1f} s; numpy "
                      "BLAS threads as configured)"}


# ---------------------------------------------------------- f-gram discovery
def bench_discover(args, world, rank, local):
    """Algorithm 3 by K-1 counting scans over a corpus resident in HBM: one
    step is one whole scone_fgram_discover call (counting scans, selection,
    list emission)."""
    import torch

    import synth
    import paper_2502_01637_gb300 as scone

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = workload(args.workload)
    n = w.B * w.L
    S = w.n_fgrams
    t0 = time.time()
    tok_np = synth.query_tokens(w)
    # the corpus in pinned host memory from scone_host_alloc (a huge-page
    # mapping): torch's pin_memory buffers (small pages) copied in at 15-112
    # GB/s on some calls instead of 211, from address translation of the pages
    host_buf = scone.scone_host_alloc(tok_np.nbytes)
    host_np = host_buf.numpy(np.int32)[:tok_np.size].reshape(tok_np.shape)
    host_np[:] = tok_np
    host_tok = torch.from_numpy(host_np)
    tok = host_tok.to(dev)
    out_tok = torch.empty((S, w.K), dtype=torch.int32, device=dev)
    out_len = torch.empty(S, dtype=torch.uint8, device=dev)
    out_cnt = torch.empty(S, dtype=torch.int32, device=dev)
    ws = scone.scone_discover_create()
    setup_s = time.time() - t0
    stream = torch.cuda.current_stream()

    def step(src):
        return scone.scone_fgram_discover(src, w.vocab, w.K, S, w.min_count, out_tok, out_len,
                                          out_cnt, workspace=ws)

    for _ in range(args.warmup):
        step(tok)
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    stats = []
    clocks = ClockSampler(local)
    barrier(world)
    with clocks:
        for k in range(args.steps):
            ev[k][0].record(stream)
            stats.append(step(tok)[3])
            ev[k][1].record(stream)
        torch.cuda.synchronize()
    barrier(world)
    ms = max_over_ranks(statistics.mean(a.elapsed_time(b) for a, b in ev), world)
    st = stats[-1]

    # end to end: corpus from pinned host memory, the call, the list back to the host
    out_bufs = [scone.scone_host_alloc(t.numel() * t.element_size()) for t in (out_tok, out_len, out_cnt)]
    host_out = [torch.from_numpy(b.numpy(np.uint8)[:t.numel() * t.element_size()]).view(t.dtype)
                .reshape(t.shape) for b, t in zip(out_bufs, (out_tok, out_len, out_cnt))]
    e2e_t, e2e_h2d = [], []
    for k in range(max(2, min(args.steps, 5))):
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t1 = time.perf_counter()
        e0.record(stream)
        tok.copy_(host_tok, non_blocking=True)
        e1.record(stream)
        ft, fl, fc, _ = step(tok)
        m = fl.shape[0]
        for h, d in zip(host_out, (ft, fl, fc)):
            h[:m].copy_(d, non_blocking=True)
        torch.cuda.synchronize()
        e2e_t.append(time.perf_counter() - t1)
        e2e_h2d.append(e0.elapsed_time(e1))
    e2e_ms = max_over_ranks(1e3 * statistics.mean(e2e_t), world)
    m = int(st["frequent"][2] + sum(st["frequent"][3:]))
    n_sel = min(S, m)

    # roofline of the dominant kernel: the counting pass of scan 2 (bincount_kernel).
    # Algorithmic bytes: each binned window's record (8-byte key + 2-byte
    # offset) read once, the per-chunk bin offsets read once, and each distinct
    # key's 16-byte slot brought from DRAM and written back as one 32-byte
    # sector each way.
    ms_count = statistics.mean(s_["ms_count"][2] for s_ in stats)
    n_chunks = -(-n // 16384)
    bytes_count = 10 * st["flushes"][2] + 4 * 1025 * n_chunks + 64 * st["distinct"][2]
    hbm, peak_src = measured_peaks()
    achieved = bytes_count / (ms_count * 1e-3) / 1e9
    res = {
        "metric": METRIC_DISCOVER,
        "value": world * n / (ms * 1e-3),
        "unit": "corpus tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "int32",
        "data": "synthetic corpus (seeded Zipf(1.1) sequences over 1e5 token ids)",
        "config": {"workload": (f"{w.name}: f-grams of length 2..{w.K} with count >= "
                                f"{w.min_count}, the {S} most frequent, from {w.B} x {w.L} = "
                                f"{n} corpus tokens in HBM"),
                   "l2": "corpus (4.3 GB) and counting table far larger than L2; no flush",
                   "timing": "CUDA events around each whole scone_fgram_discover call"},
        "roofline": {
            "bound": "hbm",
            "achieved": achieved,
            "peak": hbm,
            "unit": "GB/s",
            "frac": achieved / hbm,
            "traffic": (profiled_traffic(w.name, "bincount_kernel", DISCOVER_SOURCES)
                        if w.name == "discover" else None),
            "peak_source": peak_src,
            "algorithmic_bytes_per_launch": bytes_count,
            "kernel": ("bincount_kernel of scan 2 (10 B per binned window + 4 B per chunk and "
                       "bin + 64 B per distinct key; bound in practice by L2 atomics on the "
                       "resident table region, not by DRAM)"),
            "kernel_ms": ms_count,
            "kernel_share_of_step": ms_count / ms,
        },
        "e2e": {"value": world * n / (e2e_ms * 1e-3), "unit": "corpus tokens/s",
                "h2d_bytes_per_step": 4 * n,
                "d2h_bytes_per_step": n_sel * (4 * w.K + 1 + 4),
                "what": "pinned corpus -> device, scone_fgram_discover, f-gram list -> "
                        "pinned host",
                "per_call_ms": [round(1e3 * x, 2) for x in e2e_t],
                "corpus_h2d_ms": [round(x, 2) for x in e2e_h2d],
                "spread": max(e2e_t) / min(e2e_t) - 1.0},
        # per call: bin, hotflush, bincount, flagbin, unsort, scan and assign
        # per scan; then 4 radix-select histograms (only when the cut falls
        # inside the list), select_count, two scans and emit
        "gpu_launches": args.steps * (7 * (w.K - 1) + (8 if S < m else 4)),
        "clocks": clocks.summary(),
        "discover": {k: st[k] for k in ("candidates", "distinct", "frequent", "flushes",
                                         "threshold", "selected_at_threshold",
                                         "table_bytes_max", "ms_bin", "ms_count", "ms_flag",
                                         "ms_scan",
                                         "ms_select", "ms_total", "ms_alloc_host",
                                         "workspace_bytes")},
        "setup_s": setup_s,
    }
    if rank == 0 and not args.no_cpu_baseline:
        res["cpu_baseline"] = cpu_baseline_discover(w, tok_np)
    ws.close()
    return res


def cpu_baseline_discover(w, tok, budget_s: float = 10.0):
    """The discovery oracle (single thread, std::map of every n-gram) on a
    bounded prefix of the same corpus, grown until it takes about budget_s."""
    import oracle

    seqs = 64
    while True:
        t0 = time.perf_counter()
        oracle.discover(tok[:seqs], w.K, w.vocab, w.n_fgrams, w.min_count)
        dt = time.perf_counter() - t0
        if dt >= budget_s / 3 or seqs >= tok.shape[0]:
            break
        seqs *= 2
    return {"value": seqs * w.L / dt, "unit": "corpus tokens/s", "cores": 1, "kind": "oracle",
            "sample": f"oracle discovery over the first {seqs} x {w.L} tokens of the corpus "
                      f"({dt:.1f} s)"}


# ----------------------------------------------------------- reference arm
PREFILL_WORKLOADS = ("tiny", "prefill_1b", "large_hbm", "stress_k5", "prefill_profile",
                     "large_hbm_profile", "stress_profile")


def bench_reference(args, world, rank):
    """The reference arm: the CPU oracle (the plain definition of Algorithm 1,
    single-threaded) on the host cores, on the measured arm's config, metric
    and unit. Each step embeds one whole batch of the workload (B x L
    tokens), rotating over the same batches the measured arm times."""
    import synth
    import oracle

    w = workload(args.workload)
    if args.workload not in PREFILL_WORKLOADS:
        return {"impl": "reference", "unavailable": (
            f"the reference arm times the embedding oracle on the prefill workloads; "
            f"{args.workload} reports its CPU oracle under cpu_baseline of its own line")}
    t0 = time.time()
    fg_tok, fg_len, _ = synth.fgram_set(w)
    # batch k of rank r is the one the measured arm's rank r embeds at step k
    batches = [[synth.query_tokens(w, range((r * N_BATCHES + k) * w.B,
                                            (r * N_BATCHES + k + 1) * w.B))
                for k in range(N_BATCHES)] for r in range(world)]
    o = oracle.Oracle(fg_tok, fg_len, w.K, w.vocab)
    # rows the batches select, generated on the host; T in full
    F = host_F_for(o, [b for per_rank in batches for b in per_rank], w)
    T = synth.rows_range_cpu(synth.T_seed(w), w.d, 0, w.vocab)
    setup_s = time.time() - t0

    def step(k):
        for per_rank in batches:                     # the whole job's batch of step k
            o.embed(per_rank[k % N_BATCHES], F, T)

    for k in range(args.warmup):
        step(k)
    times = []
    for k in range(args.steps):
        t1 = time.perf_counter()
        step(k)
        times.append(time.perf_counter() - t1)
    ms = 1e3 * statistics.mean(times)
    n_tok = world * w.B * w.L
    val = n_tok / (ms * 1e-3)
    sample = (f"each step: the oracle over the whole job's batch of {w.name} ({world} x "
              f"{w.B} x {w.L} = {n_tok} tokens; {N_BATCHES} batches per rank in rotation; "
              f"map build untimed)")
    return {
        "impl": "reference", "metric": METRIC, "value": val, "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded Zipf token streams and f-gram sets, N(0,0.02)-like bf16 rows)",
        "config": {**prefill_config(w, world),
                   "timing": "host clock around the oracle calls of one step (the whole "
                             "job's batch)"},
        "cpu_baseline": {"value": val, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": val, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        "setup_s": setup_s,
    }


EXTRA_KEYS = ("value", "unit", "ms_per_step", "steps", "warmup", "config", "roofline", "e2e",
              "gpu_launches", "clocks", "match_rate", "match_len_hist", "kernel_ms_median",
              "replay_frac")


def extra_summary(res: dict) -> dict:
    """The keys of another workload's line that go under 'extra' of the main one."""
    out = {k: res[k] for k in EXTRA_KEYS if k in res}
    if "roofline" in out:
        out["roofline"] = {k: v for k, v in out["roofline"].items()}
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="scone", choices=["scone", "reference"])
    ap.add_argument("--workload", default=None,
                    choices=["tiny", "prefill_1b", "large_hbm", "stress_k5", "prefill_profile",
                             "large_hbm_profile", "stress_profile",
                             "offload_decode", "offload_decode_first_seen", "decode_profile",
                             "prescan", "discover", "discover_k5", "discover_profile",
                             "mixed_serving", "precompute", "gemm_profile", "store_decode"],
                    help="default: large_hbm, plus prefill_1b and offload_decode under "
                         "'extra' (single GPU)")
    ap.add_argument("--no-extras", action="store_true",
                    help="without --workload: measure large_hbm only")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--load-factor", type=float, default=None,
                    help="prefill workloads: the table's load factor (default: the workload's)")
    ap.add_argument("--copy", default="auto",
                    choices=["auto", "registers", "bulk", "split", "pipelined"],
                    help="row copy method of the fused kernel (results are identical)")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)
    extras = args.workload is None and not args.no_extras
    if args.workload is None:
        args.workload = DEFAULT_WORKLOAD
    world, rank, local = dist_setup()
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(bench_reference(args, world, rank)), flush=True)
        return
    import __graft_entry__

    if rank == 0:
        __graft_entry__.build()
    barrier(world)
    if args.workload in ("offload_decode", "offload_decode_first_seen", "decode_profile"):
        res = bench_decode(args, world, rank, local)
    elif args.workload == "prescan":
        res = bench_prescan(args, world, rank, local)
    elif args.workload == "mixed_serving":
        res = bench_mixed(args, world, rank, local)
    elif args.workload == "precompute":
        res = bench_precompute(args, world, rank, local)
    elif args.workload == "gemm_profile":
        res = bench_gemm(args, world, rank, local)
    elif args.workload == "store_decode":
        res = bench_store(args, world, rank, local)
    elif args.workload in ("discover", "discover_k5", "discover_profile"):
        res = bench_discover(args, world, rank, local)
    else:
        res = bench_prefill(args, world, rank, local)
    if extras and world == 1:
        # the other two configurations measured in the same process: the
        # 1B-model prefill and the offloaded tier (F in host memory, read over
        # the host link), each with its own roofline, clocks and e2e
        import torch

        res["extra"] = {}
        for name, fn in (("prefill_1b", bench_prefill), ("offload_decode", bench_decode)):
            torch.cuda.empty_cache()
            sub = argparse.Namespace(**vars(args))
            sub.workload = name
            sub.no_cpu_baseline = True
            sub.steps = max(args.steps, 200)
            sub.warmup = max(args.warmup, 10)
            res["extra"][name] = extra_summary(fn(sub, world, rank, local))
            res["gpu_launches_extra"] = res.get("gpu_launches_extra", 0) + \
                res["extra"][name]["gpu_launches"]
    if rank == 0:
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()
