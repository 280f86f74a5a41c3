// Fused embed with the match of the next tile interleaved into the copy of
// the current one (SCONE_COPY_PIPELINED).
//
// Same selection and output as embed_kernel (Algorithm 1, inference branch,
// Sec. 3), same work split (a persistent grid, the flattened positions split
// evenly over its warps, tiles of 32 positions, one lane per position). In
// embed_kernel a warp matches a tile, then copies its rows, then matches the
// next tile: the match is a chain of dependent loads (window tokens, first
// buckets, second buckets) during which the warp has no row loads in flight,
// and under a saturated HBM each of those round trips takes microseconds.
//
// Here the match of tile i+1 is cut at those dependent loads into four
// stages, and the copy of tile i into four segments of chunks; stage k of the
// next tile runs after segment k of the current copy. Each stage issues its
// loads and leaves them in flight while the warp copies the next segment, so
// the match latency hides behind row traffic and the warp keeps its row
// loads in flight nearly all the time. The first tile of a warp is matched
// before its copy starts; the match steps and their order are those of
// match_position (scone_device.cuh), split where a stage waits on a load.
//
// The buckets a stage loads go to shared memory with cp.async, so the state
// that lives across a copy segment is the window tokens and a few flags and
// the copy keeps as many loads in flight as embed_kernel does. Used for the
// 16-byte-aligned case with 16-byte slots (FMT16) and K <= 5; other calls
// take embed_kernel.
//
// On a table with a suffix index (scone_device.cuh) the match walks the
// lengths instead: n = 2, 3, ... one bucket at a time, stopping at the first
// window that is absent or has no extension bit. The K-1 first buckets of a
// position are mostly distinct cold sectors, and random sectors cost far
// more DRAM time than their bytes; the walk reads about 1.7 lookups per
// position on Zipf text at K = 5 instead of K-1. It takes more dependent
// round trips, so a round runs after every chunk of the copy (one chunk is
// one batch of row loads in flight), and rounds left when the copy ends run
// back to back. The walk ends at the same longest f-gram: every suffix of
// that f-gram is present with its extension bit, and no window longer than
// an absent or unextended one can be an f-gram.

#include "scone_host.h"
#include "scone_walk.cuh"

namespace scone {

constexpr int kPipeThreads = 256;
constexpr int kPipeWarps = kPipeThreads / 32;

namespace {

template <int KT>
struct PipeTuning {
  static constexpr int kLoads = KT <= 3 ? 8 : 16;        // 16-byte loads in flight per lane
  static constexpr int kMinBlocks = KT <= 3 ? 3 : 2;
};

// The match of one position (16-byte slots), in four stages that each end
// with loads issued: the window tokens into registers, the buckets into this
// lane's shared-memory slots `sb` (one per length).
template <int KT>
struct PipeMatch {
  int32_t w[KT];              // window tokens, newest first
  int32_t r1[KT - 1];
  int nmax;                   // longest usable window
  uint32_t second;            // bit n-2: length n needs its second bucket
  bool active, bad;
  Bucket* sb;                 // [KT - 1] bucket of each length (first, then second)

  // stage 0: the window tokens (loads issued)
  __device__ __forceinline__ void stage0(const TableView& t, const int32_t* __restrict__ tok,
                                         int64_t p, int32_t i, bool act) {
    active = act;
    bad = false;
    nmax = 0;
    second = 0;
    if (!act) return;
    w[0] = __ldg(tok + p);
    nmax = t.K < i + 1 ? t.K : i + 1;
#pragma unroll
    for (int j = 1; j < KT; ++j) w[j] = (j < nmax) ? __ldg(tok + p - j) : 0;
  }
  // stage 1: validity, keys, and the first bucket of every usable length
  __device__ __forceinline__ void stage1(const TableView& t) {
    if (!active) return;
    if (!valid_token(w[0], t.vocab)) {
      bad = true;
      return;
    }
    int nvalid = 1;
#pragma unroll
    for (int j = 1; j < KT; ++j)
      if (nvalid == j && j < nmax && valid_token(w[j], t.vocab)) nvalid = j + 1;
    nmax = nvalid;
#pragma unroll
    for (int n = 2; n <= KT; ++n) {
      if (n <= nmax) {
        uint64_t b1, b2;
        cuckoo_buckets(key_hash<FMT16>(window_key<FMT16, KT>(w, n, t.bits), t.hash_seed),
                       t.n_buckets, &b1, &b2);
        bucket_async(&sb[n - 2], t, b1);
      }
    }
    cp_async_commit();
  }
  // stage 2: first-round hits; the second buckets still needed (loads issued)
  __device__ __forceinline__ void stage2(const TableView& t) {
    second = 0;
    if (!active || bad) return;
    cp_async_wait_all();
#pragma unroll
    for (int n = 2; n <= KT; ++n) {
      r1[n - 2] = -1;
      if (n <= nmax) {
        BucketData<FMT16> v;
        v.part[0] = sb[n - 2];
        r1[n - 2] = find_in_bucket<FMT16>(v, window_key<FMT16, KT>(w, n, t.bits));
        if (r1[n - 2] < 0 && bucket_full<FMT16>(v)) second |= 1u << (n - 2);
      }
    }
    // only lengths longer than the longest first-round hit matter
    int best = 0;
#pragma unroll
    for (int n = 2; n <= KT; ++n)
      if (r1[n - 2] >= 0) best = n;
    second &= ~((1u << (best > 1 ? best - 1 : 0)) - 1u);
    if (second && t.probe_limit >= 2) {
#pragma unroll
      for (int n = 2; n <= KT; ++n) {
        if (second & (1u << (n - 2))) {
          uint64_t b1, b2;
          cuckoo_buckets(key_hash<FMT16>(window_key<FMT16, KT>(w, n, t.bits), t.hash_seed),
                         t.n_buckets, &b1, &b2);
          bucket_async(&sb[n - 2], t, b2);
        }
      }
      cp_async_commit();
    }
  }
  // stage 3: the longest hit. Returns the row (or -1), sets *len and *err as
  // match_position does.
  __device__ __forceinline__ int32_t stage3(const TableView& t, int* len, int* err) {
    if (bad) {
      *err = SCONE_ERR_TOKEN_RANGE;
      *len = 0;
      return -1;
    }
    if (second) {
      if (t.probe_limit < 2) {
        *err = SCONE_ERR_PROBE_LIMIT;
        *len = 0;
        return -1;
      }
      cp_async_wait_all();
#pragma unroll
      for (int n = 2; n <= KT; ++n) {
        if (second & (1u << (n - 2))) {
          BucketData<FMT16> v;
          v.part[0] = sb[n - 2];
          r1[n - 2] = find_in_bucket<FMT16>(v, window_key<FMT16, KT>(w, n, t.bits));
        }
      }
    }
#pragma unroll
    for (int n = KT; n >= 2; --n) {
      if (n <= nmax && r1[n - 2] >= 0) {
        *len = n;
        return r1[n - 2];
      }
    }
    *len = 1;
    return -1;
  }
};

template <int KT>
__device__ __forceinline__ const uint4* pipe_finish(const TableView& t, PipeMatch<KT>& m,
                                                    int64_t p, int32_t* __restrict__ row_out,
                                                    uint8_t* __restrict__ len_out) {
  if (!m.active) return nullptr;
  int len = 0, err = 0;
  const int32_t r = m.stage3(t, &len, &err);
  if (row_out) row_out[p] = r;
  if (len_out) len_out[p] = (uint8_t)len;
  if (err) {
    record_error(t, err);
    return nullptr;
  }
  return reinterpret_cast<const uint4*>(r >= 0 ? t.F + (int64_t)r * t.d
                                               : t.T + (int64_t)m.w[0] * t.d);
}

// The walk variant of the kernel below: same tiles, copies and output.
template <int KT>
__global__ void __launch_bounds__(kPipeThreads, kWalkMinBlocks)
    embed_walk_kernel(const TableView t, const int32_t* __restrict__ tok, int64_t n_tok,
                      int32_t L, uint8_t* __restrict__ out, int32_t* __restrict__ row_out,
                      uint8_t* __restrict__ len_out) {
  constexpr int U = kWalkLoads;
  __shared__ const uint4* src_s[kPipeWarps][2][32];
  __shared__ __align__(16) Bucket bucket_s[kPipeWarps][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int epr = t.d >> 3;                      // 16-byte elements per row
  const int64_t nw = (int64_t)gridDim.x * kPipeWarps;
  const int64_t wid = (int64_t)blockIdx.x * kPipeWarps + warp;
  const int64_t lo = n_tok * wid / nw, hi = n_tok * (wid + 1) / nw;
  if (lo >= hi) return;
  PipeWalk<KT> m;
  m.sb = &bucket_s[warp][lane];
  int buf = 0;
  int64_t base = lo;
  int nrows = (int)(hi - base < kWalkFirst ? hi - base : kWalkFirst);
  {  // the warp's first tile: its rounds back to back
    const int64_t p = base + lane;
    m.start(t, tok, p, (int32_t)(p % L), lane < nrows);
    while (__any_sync(0xFFFFFFFFu, m.state != 0)) m.round(t);
    src_s[warp][buf][lane] = lane < nrows ? walk_finish<KT>(t, m, p, row_out, len_out) : nullptr;
    __syncwarp();
  }
  while (base < hi) {
    const int64_t nbase = base + nrows;
    const int nn = nbase < hi ? (int)(hi - nbase < 32 ? hi - nbase : 32) : 0;
    const int64_t np = nbase + lane;
    const int64_t total = (int64_t)nrows * epr;
    const int nchunks = (int)((total + 32 * U - 1) / (32 * U));
    const uint4* const* src = src_s[warp][buf];
    uint4* dst = reinterpret_cast<uint4*>(out) + base * epr;
    int r = 0, col = lane;
    while (col >= epr) {
      col -= epr;
      ++r;
    }
    if (nn) m.start(t, tok, np, (int32_t)(np % L), lane < nn);
    for (int c = 0; c < nchunks; ++c) {
      copy_chunks<U>(src, dst, nrows, epr, total, lane, c, c + 1, r, col);
      if (nn) m.round(t);
    }
    if (nn) {
      while (__any_sync(0xFFFFFFFFu, m.state != 0)) m.round(t);
      src_s[warp][buf ^ 1][lane] = lane < nn ? walk_finish<KT>(t, m, np, row_out, len_out)
                                             : nullptr;
    }
    __syncwarp();
    buf ^= 1;
    base = nbase;
    nrows = nn;
  }
}

template <int KT>
__global__ void __launch_bounds__(kPipeThreads, PipeTuning<KT>::kMinBlocks)
    embed_pipe_kernel(const TableView t, const int32_t* __restrict__ tok, int64_t n_tok,
                      int32_t L, uint8_t* __restrict__ out, int32_t* __restrict__ row_out,
                      uint8_t* __restrict__ len_out) {
  constexpr int U = PipeTuning<KT>::kLoads;
  __shared__ const uint4* src_s[kPipeWarps][2][32];
  __shared__ __align__(16) Bucket bucket_s[kPipeWarps][32][KT - 1];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int epr = t.d >> 3;                      // 16-byte elements per row
  const int64_t nw = (int64_t)gridDim.x * kPipeWarps;
  const int64_t wid = (int64_t)blockIdx.x * kPipeWarps + warp;
  const int64_t lo = n_tok * wid / nw, hi = n_tok * (wid + 1) / nw;
  if (lo >= hi) return;
  PipeMatch<KT> m;
  m.sb = bucket_s[warp][lane];
  int buf = 0;
  int64_t base = lo;
  int nrows = (int)(hi - base < 32 ? hi - base : 32);
  {  // the warp's first tile: its stages back to back
    const int64_t p = base + lane;
    m.stage0(t, tok, p, (int32_t)(p % L), lane < nrows);
    m.stage1(t);
    m.stage2(t);
    src_s[warp][buf][lane] = pipe_finish<KT>(t, m, p, row_out, len_out);
    __syncwarp();
  }
  while (base < hi) {
    const int64_t nbase = base + 32;
    const int nn = nbase < hi ? (int)(hi - nbase < 32 ? hi - nbase : 32) : 0;
    const int64_t np = nbase + lane;
    const int64_t total = (int64_t)nrows * epr;
    const int nchunks = (int)((total + 32 * U - 1) / (32 * U));
    const int c1 = nchunks / 4, c2 = nchunks / 2, c3 = (3 * nchunks) / 4;
    const uint4* const* src = src_s[warp][buf];
    uint4* dst = reinterpret_cast<uint4*>(out) + base * epr;
    int r = 0, col = lane;
    while (col >= epr) {
      col -= epr;
      ++r;
    }
    copy_chunks<U>(src, dst, nrows, epr, total, lane, 0, c1, r, col);
    if (nn) m.stage0(t, tok, np, (int32_t)(np % L), lane < nn);
    copy_chunks<U>(src, dst, nrows, epr, total, lane, c1, c2, r, col);
    if (nn) m.stage1(t);
    copy_chunks<U>(src, dst, nrows, epr, total, lane, c2, c3, r, col);
    if (nn) m.stage2(t);
    copy_chunks<U>(src, dst, nrows, epr, total, lane, c3, nchunks, r, col);
    if (nn) src_s[warp][buf ^ 1][lane] = pipe_finish<KT>(t, m, np, row_out, len_out);
    __syncwarp();
    buf ^= 1;
    base = nbase;
    nrows = nn;
  }
}

using PipeFn = void (*)(TableView, const int32_t*, int64_t, int32_t, uint8_t*, int32_t*,
                        uint8_t*);

}  // namespace

bool pipe_eligible(const scone_table* tb, const void* out) {
  return tb->fmt == FMT16 && tb->view.K <= 5 && row_copy_width(tb->view, out) == 16;
}

int launch_embed_pipe(const scone_table* tb, const int32_t* tok, int64_t n, int32_t L,
                      uint8_t* out, int32_t* row, uint8_t* len, cudaStream_t stream) {
  // the walk needs the suffix index; with a one-bucket probe limit (a
  // diagnostic) the staged match reports errors where embed_kernel does
  const bool walk = tb->view.suffix_index && tb->view.probe_limit >= 2;
  const PipeFn fn = walk ? (tb->view.K <= 3 ? embed_walk_kernel<3> : embed_walk_kernel<5>)
                         : (tb->view.K <= 3 ? embed_pipe_kernel<3> : embed_pipe_kernel<5>);
  // every resident block, unless warps would get fewer than 8 rows each
  const int64_t cap = (int64_t)sm_count() * blocks_per_sm((const void*)fn, kPipeThreads, 0);
  const int64_t need = (n + kPipeWarps * 8 - 1) / (kPipeWarps * 8);
  const int grid = (int)(need < cap ? (need < 1 ? 1 : need) : cap);
  fn<<<grid, kPipeThreads, 0, stream>>>(tb->view, tok, n, L, out, row, len);
  return cudaGetLastError() == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}

}  // namespace scone
