// Prefill path: match, gather and the fused embed (Algorithm 1, inference
// branch, Sec. 3), plus the launch helpers.
//
// Work split: the grid is persistent (as many 8-warp blocks as are resident
// at once, all SMs equally loaded) and the flattened [B x L] positions are
// split evenly over all its warps, so every warp moves the same number of
// rows (+-1). A warp walks its range in tiles of up to 32 positions: each
// lane matches one position (the first buckets of all K-1 candidate lengths
// read at once, then the second buckets still needed; longest hit kept), the
// selected row addresses go to shared memory, and the warp then streams the
// rows to the contiguous output block with 16-byte loads and streaming
// (evict-first) stores.
//
// Occupancy: the match of a tile is a chain of dependent loads during which
// its warp moves no rows, so the kernel wants many resident warps; the copy
// wants many loads in flight per warp. For K <= 3 the best measured split is
// 8 loads in flight per lane with 3 blocks (24 warps) per SM (80 registers,
// no spills); for the longer unrolls 16 loads in flight with 2 blocks
// (K <= 5) or 1 block (K <= 8), where the keys need more registers.

#include <map>
#include <mutex>
#include <utility>

#include "scone_host.h"
#include "scone_walk.cuh"

namespace scone {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

int sm_count() {
  int dev = 0, sms = 1;
  cudaGetDevice(&dev);
  static std::mutex mu;
  static std::map<int, int> cache;
  std::lock_guard<std::mutex> lk(mu);
  auto it = cache.find(dev);
  if (it != cache.end()) return it->second;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cache[dev] = sms;
  return sms;
}

int blocks_per_sm(const void* fn, int threads, size_t smem) {
  int dev = 0;
  cudaGetDevice(&dev);
  static std::mutex mu;
  static std::map<std::pair<const void*, int>, int> cache;
  std::lock_guard<std::mutex> lk(mu);
  const auto key = std::make_pair(fn, dev * 4096 + threads);
  auto it = cache.find(key);
  if (it != cache.end()) return it->second;
  int n = 1;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, threads, smem) != cudaSuccess ||
      n < 1) {
    cudaGetLastError();
    n = 1;
  }
  cache[key] = n;
  return n;
}

namespace {

int grid_size(const void* fn, int64_t blocks_needed) {
  const int64_t cap = (int64_t)sm_count() * blocks_per_sm(fn, kThreads, 0);
  int64_t g = blocks_needed < cap ? blocks_needed : cap;
  return g < 1 ? 1 : (int)g;
}

// Copy kernels: every resident block, unless the batch is so small that
// warps would get fewer than kMinRowsPerWarp rows each.
constexpr int64_t kMinRowsPerWarp = 8;
int copy_grid(const void* fn, int64_t n_tok) {
  return grid_size(fn, (n_tok + kWarps * kMinRowsPerWarp - 1) / (kWarps * kMinRowsPerWarp));
}

__device__ __forceinline__ int32_t pos_in_seq(int64_t p, int32_t L) { return (int32_t)(p % L); }

template <int FMT, int KT>
__global__ void __launch_bounds__(kThreads)
    match_kernel(const TableView t, const int32_t* __restrict__ tok, int64_t n_tok, int32_t L,
                 int32_t* __restrict__ row_out, uint8_t* __restrict__ len_out) {
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < n_tok;
       p += (int64_t)gridDim.x * blockDim.x) {
    const int32_t x = __ldg(tok + p);
    int len = 0, err = 0;
    const int32_t r = match_position<FMT, KT>(t, tok, p, pos_in_seq(p, L), x, &len, &err);
    if (err) record_error(t, err);
    row_out[p] = r;
    if (len_out) len_out[p] = (uint8_t)len;
  }
}

// match_kernel with the walk over the suffix index (tables that have one).
template <int KT>
__global__ void __launch_bounds__(kThreads)
    match_walk_kernel(const TableView t, const int32_t* __restrict__ tok, int64_t n_tok,
                      int32_t L, int32_t* __restrict__ row_out, uint8_t* __restrict__ len_out) {
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < n_tok;
       p += (int64_t)gridDim.x * blockDim.x) {
    const int32_t x = __ldg(tok + p);
    int len = 0, err = 0;
    const int32_t r = walk_position<KT>(t, tok, p, pos_in_seq(p, L), x, &len, &err);
    if (err) record_error(t, err);
    row_out[p] = r;
    if (len_out) len_out[p] = (uint8_t)len;
  }
}

// Positions [lo, hi) of warp w out of nw, an even split of n.
__device__ __forceinline__ void warp_range(int64_t n, int64_t w, int64_t nw, int64_t* lo,
                                           int64_t* hi) {
  *lo = n * w / nw;
  *hi = n * (w + 1) / nw;
}

template <int KT>
struct EmbedTuning {
  static constexpr int kLoads = KT <= 3 ? 8 : 16;
  static constexpr int kMinBlocks = KT <= 3 ? 3 : (KT <= 5 ? 2 : 1);
};

template <int FMT, int KT, int W>
__global__ void __launch_bounds__(kThreads, EmbedTuning<KT>::kMinBlocks)
    embed_kernel(const TableView t, const int32_t* __restrict__ tok, int64_t n_tok, int32_t L,
                 uint8_t* __restrict__ out, int32_t* __restrict__ row_out,
                 uint8_t* __restrict__ len_out, int width) {
  __shared__ const void* src_s[kWarps][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int row_bytes = t.d * 2;
  int64_t lo, hi;
  warp_range(n_tok, (int64_t)blockIdx.x * kWarps + warp, (int64_t)gridDim.x * kWarps, &lo, &hi);
  for (int64_t base = lo; base < hi; base += 32) {
    const int nrows = (int)(hi - base < 32 ? hi - base : 32);
    const int64_t p = base + lane;
    const void* src = nullptr;
    if (lane < nrows) {
      const int32_t x = __ldg(tok + p);
      int len = 0, err = 0;
      const int32_t r = match_position<FMT, KT>(t, tok, p, pos_in_seq(p, L), x, &len, &err);
      if (err) {
        record_error(t, err);
      } else {
        src = r >= 0 ? static_cast<const void*>(t.F + (int64_t)r * t.d)
                     : static_cast<const void*>(t.T + (int64_t)x * t.d);
      }
      if (row_out) row_out[p] = r;
      if (len_out) len_out[p] = (uint8_t)len;
    }
    src_s[warp][lane] = src;
    __syncwarp();
    warp_copy_rows_w<W, EmbedTuning<KT>::kLoads>(src_s[warp], out + base * (int64_t)row_bytes,
                                                 nrows, row_bytes, width, lane);
    __syncwarp();
  }
}

template <int W>
__global__ void __launch_bounds__(kThreads)
    gather_kernel(const TableView t, const int32_t* __restrict__ tok,
                  const int32_t* __restrict__ row, int64_t n_tok, uint8_t* __restrict__ out,
                  int width) {
  __shared__ const void* src_s[kWarps][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int row_bytes = t.d * 2;
  int64_t lo, hi;
  warp_range(n_tok, (int64_t)blockIdx.x * kWarps + warp, (int64_t)gridDim.x * kWarps, &lo, &hi);
  for (int64_t base = lo; base < hi; base += 32) {
    const int nrows = (int)(hi - base < 32 ? hi - base : 32);
    const int64_t p = base + lane;
    const void* src = nullptr;
    if (lane < nrows) {
      const int32_t r = __ldg(row + p);
      if (r >= 0) {
        if (r < t.n_fgrams) src = t.F + (int64_t)r * t.d;
        else record_error(t, SCONE_ERR_INVALID_ARG);
      } else {
        const int32_t x = __ldg(tok + p);
        if (valid_token(x, t.vocab)) src = t.T + (int64_t)x * t.d;
        else record_error(t, SCONE_ERR_TOKEN_RANGE);
      }
    }
    src_s[warp][lane] = src;
    __syncwarp();
    warp_copy_rows_w<W>(src_s[warp], out + base * (int64_t)row_bytes, nrows, row_bytes, width,
                        lane);
    __syncwarp();
  }
}

using MatchFn = void (*)(TableView, const int32_t*, int64_t, int32_t, int32_t*, uint8_t*);
using EmbedFn = void (*)(TableView, const int32_t*, int64_t, int32_t, uint8_t*, int32_t*,
                         uint8_t*, int);

// K <= 3 -> unrolled for 3, K <= 5 -> 5, else 8. The 32-byte key format only
// arises for K*b > 92, so it is instantiated for the two larger unrolls.
MatchFn pick_match(int fmt, int K) {
  if (fmt == FMT16) {
    if (K <= 3) return match_kernel<FMT16, 3>;
    if (K <= 5) return match_kernel<FMT16, 5>;
    return match_kernel<FMT16, 8>;
  }
  if (K <= 5) return match_kernel<FMT32, 5>;
  return match_kernel<FMT32, 8>;
}

template <int W>
EmbedFn pick_embed_w(int fmt, int K) {
  if (fmt == FMT16) {
    if (K <= 3) return embed_kernel<FMT16, 3, W>;
    if (K <= 5) return embed_kernel<FMT16, 5, W>;
    return embed_kernel<FMT16, 8, W>;
  }
  if (K <= 5) return embed_kernel<FMT32, 5, W>;
  return embed_kernel<FMT32, 8, W>;
}

EmbedFn pick_embed(int fmt, int K, int width) {
  return width == 16 ? pick_embed_w<16>(fmt, K) : pick_embed_w<0>(fmt, K);
}

bool misaligned(const void* p, uintptr_t a) { return ((uintptr_t)p & (a - 1)) != 0; }

// Whether p is host memory (mapped pinned memory read over the host link).
bool is_host_memory(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeHost;
}

}  // namespace

}  // namespace scone

using namespace scone;

extern "C" int scone_match(const scone_table* tb, const int32_t* tok, int32_t B, int32_t L,
                           int32_t* row, uint8_t* len, void* stream) {
  if (!tb || B < 0 || L < 0) return SCONE_ERR_INVALID_ARG;
  const int64_t n = (int64_t)B * L;
  if (n == 0) return SCONE_OK;
  if (!tok || !row || misaligned(tok, 4) || misaligned(row, 4)) return SCONE_ERR_INVALID_ARG;
  DeviceGuard g(tb->device);
  // the walk over the suffix index where the table has one and the tokens are
  // in device memory (REGISTERS keeps the lookups of every length; the walk
  // assumes the default probe limit). Over the host link the walk's longer
  // chain of dependent reads per position costs more than its fewer bucket
  // sectors save: on a 1.07e9-token corpus in host memory 40.0 ms against
  // 37.9 for the all-length lookups, in HBM 28.3 against 34.1.
  const bool walk = tb->view.suffix_index && tb->view.probe_limit >= 2 && tb->fmt == FMT16 &&
                    tb->view.K <= 5 && tb->copy_mode != SCONE_COPY_REGISTERS &&
                    !is_host_memory(tok);
  const MatchFn fn = walk ? (tb->view.K <= 3 ? match_walk_kernel<3> : match_walk_kernel<5>)
                          : pick_match(tb->fmt, tb->view.K);
  const int grid = grid_size((const void*)fn, (n + kThreads - 1) / kThreads);
  fn<<<grid, kThreads, 0, (cudaStream_t)stream>>>(tb->view, tok, n, L, row, len);
  return cudaGetLastError() == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}

extern "C" int scone_embed_gather(const scone_table* tb, const int32_t* tok, const int32_t* row,
                                  int64_t n_tok, scone_bf16* out, void* stream) {
  if (!tb || n_tok < 0) return SCONE_ERR_INVALID_ARG;
  if (n_tok == 0) return SCONE_OK;
  if (!tok || !row || !out || misaligned(tok, 4) || misaligned(row, 4) || misaligned(out, 2))
    return SCONE_ERR_INVALID_ARG;
  DeviceGuard g(tb->device);
  const int width = row_copy_width(tb->view, out);
  const auto fn = width == 16 ? gather_kernel<16> : gather_kernel<0>;
  const int grid = copy_grid((const void*)fn, n_tok);
  fn<<<grid, kThreads, 0, (cudaStream_t)stream>>>(tb->view, tok, row, n_tok,
                                                  reinterpret_cast<uint8_t*>(out), width);
  return cudaGetLastError() == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}

extern "C" int scone_embed(const scone_table* tb, const int32_t* tok, int32_t B, int32_t L,
                           scone_bf16* out, int32_t* row, uint8_t* len, void* stream) {
  if (!tb || B < 0 || L < 0) return SCONE_ERR_INVALID_ARG;
  const int64_t n = (int64_t)B * L;
  if (n == 0) return SCONE_OK;
  if (!tok || !out || misaligned(tok, 4) || misaligned(out, 2) || (row && misaligned(row, 4)))
    return SCONE_ERR_INVALID_ARG;
  DeviceGuard g(tb->device);
  const bool bulk_ok = bulk_eligible(tb, out);
  if (tb->copy_mode == SCONE_COPY_BULK) {
    if (!bulk_ok) return SCONE_ERR_UNSUPPORTED;
    return launch_embed_bulk(tb, tok, n, L, reinterpret_cast<uint8_t*>(out), row, len,
                             (cudaStream_t)stream);
  }
  if (tb->copy_mode == SCONE_COPY_SPLIT)
    return launch_embed_split(tb, tok, n, L, reinterpret_cast<uint8_t*>(out), row, len,
                              (cudaStream_t)stream);
  // AUTO: the pipelined kernel where it applies and either walks the lengths
  // (tables with a suffix index: 6% faster than the register kernel on
  // stress_k5, K = 5, and 0.2-0.7% on the K = 3 workloads) or has a long
  // match to hide (3 < K <= 5: 0.5-1% faster on stress_k5 than the register
  // kernel; for K <= 3 without the index the register kernel is 0.7-1% faster)
  const bool pipe = tb->copy_mode == SCONE_COPY_PIPELINED ||
                    (tb->copy_mode == SCONE_COPY_AUTO &&
                     (tb->view.K > 3 || tb->view.suffix_index));
  if (pipe && pipe_eligible(tb, out))
    return launch_embed_pipe(tb, tok, n, L, reinterpret_cast<uint8_t*>(out), row, len,
                             (cudaStream_t)stream);
  const int width = row_copy_width(tb->view, out);
  const EmbedFn fn = pick_embed(tb->fmt, tb->view.K, width);
  const int grid = copy_grid((const void*)fn, n);
  fn<<<grid, kThreads, 0, (cudaStream_t)stream>>>(tb->view, tok, n, L,
                                                  reinterpret_cast<uint8_t*>(out), row, len,
                                                  width);
  return cudaGetLastError() == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}
