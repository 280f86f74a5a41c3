// Fused embed with separate matching and copying warps (SCONE_COPY_SPLIT).
//
// Same selection and output as embed_kernel (Algorithm 1, inference branch,
// Sec. 3). What differs is who waits for what. In embed_kernel each warp
// alternates between matching a tile of 32 positions (a chain of dependent
// loads: the window tokens, then the first buckets of all K-1 lengths, then
// the second buckets still needed) and copying the tile's rows, and it moves
// no bytes while it matches. With K = 5 that chain is long and the keys take
// registers that limit the resident warps.
//
// Here each CTA owns an even share of the positions, cut into tiles of 32,
// and its warps take one role for the whole launch:
//   * match warps (the first n_match warps): one lane per position, tile t
//     handled by match warp t mod n_match; the selected row addresses go into
//     slot t mod kSlots of a ring in shared memory;
//   * copy warps (the others): tile t copied by copy warp t mod n_copy with
//     16-byte loads (U in flight per lane) and streaming stores into the
//     contiguous output.
// Each slot has two mbarriers: `full` (the match warp arrives once the
// slot's 32 addresses are written) and `empty` (the copy warp arrives once
// it has copied the tile). A warp waits only on tiles before its own, so the
// ring always drains. Every wait is bounded: past kSplitSpinLimit polls the
// warp records SCONE_ERR_CUDA in the status word, raises the CTA's abort
// flag and returns; the others see the flag (or time out too) and return.

#include "scone_host.h"
#include "scone_ptx.cuh"

namespace scone {

constexpr int kSplitThreads = 256;
constexpr int kSplitWarps = kSplitThreads / 32;
constexpr int kSplitSlots = 16;
constexpr uint32_t kSplitSpinLimit = 1u << 22;

namespace {

template <int KT>
struct SplitTuning {
  static constexpr int kLoads = 16;                       // loads in flight per copy lane
  static constexpr int kMinBlocks = KT <= 5 ? 2 : 1;
  static constexpr int kMatchWarps = KT <= 3 ? 1 : 2;     // of kSplitWarps
};

__device__ __forceinline__ int32_t split_pos_in_seq(int64_t p, int32_t L) {
  return (int32_t)(p % L);
}

template <int FMT, int KT, int W>
__global__ void __launch_bounds__(kSplitThreads, SplitTuning<KT>::kMinBlocks)
    embed_split_kernel(const TableView t, const int32_t* __restrict__ tok, int64_t n_tok,
                       int32_t L, uint8_t* __restrict__ out, int32_t* __restrict__ row_out,
                       uint8_t* __restrict__ len_out, int width, int n_match) {
  __shared__ const void* src_s[kSplitSlots][32];
  __shared__ __align__(8) uint64_t full_bar[kSplitSlots];
  __shared__ __align__(8) uint64_t empty_bar[kSplitSlots];
  __shared__ int abort_s;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kSplitSlots; ++s) {
      mbar_init(saddr(&full_bar[s]), 1);
      mbar_init(saddr(&empty_bar[s]), 1);
    }
    abort_s = 0;
  }
  __syncthreads();
  const int row_bytes = t.d * 2;
  const int64_t lo = n_tok * blockIdx.x / gridDim.x;
  const int64_t hi = n_tok * (blockIdx.x + 1) / gridDim.x;
  const int64_t n_tiles = (hi - lo + 31) / 32;
  volatile int* abort_v = &abort_s;

  if (warp < n_match) {
    for (int64_t tile = warp; tile < n_tiles; tile += n_match) {
      const int s = (int)(tile % kSplitSlots);
      const int64_t round = tile / kSplitSlots;
      // the slot's previous tile must have been copied
      if (round > 0 &&
          !mbar_wait_bounded(saddr(&empty_bar[s]), (uint32_t)((round - 1) & 1),
                             kSplitSpinLimit)) {
        if (lane == 0) {
          record_error(t, SCONE_ERR_CUDA);
          *abort_v = 1;
        }
        return;
      }
      if (*abort_v) return;
      const int64_t base = lo + tile * 32;
      const int nrows = (int)(hi - base < 32 ? hi - base : 32);
      const int64_t p = base + lane;
      const void* src = nullptr;
      if (lane < nrows) {
        const int32_t x = __ldg(tok + p);
        int len = 0, err = 0;
        const int32_t r =
            match_position<FMT, KT>(t, tok, p, split_pos_in_seq(p, L), x, &len, &err);
        if (err) {
          record_error(t, err);
        } else {
          src = r >= 0 ? static_cast<const void*>(t.F + (int64_t)r * t.d)
                       : static_cast<const void*>(t.T + (int64_t)x * t.d);
        }
        if (row_out) row_out[p] = r;
        if (len_out) len_out[p] = (uint8_t)len;
      }
      src_s[s][lane] = src;
      __syncwarp();
      if (lane == 0) mbar_arrive(saddr(&full_bar[s]));
    }
    return;
  }

  const int n_copy = kSplitWarps - n_match;
  for (int64_t tile = warp - n_match; tile < n_tiles; tile += n_copy) {
    const int s = (int)(tile % kSplitSlots);
    const int64_t round = tile / kSplitSlots;
    if (!mbar_wait_bounded(saddr(&full_bar[s]), (uint32_t)(round & 1), kSplitSpinLimit)) {
      if (lane == 0) {
        record_error(t, SCONE_ERR_CUDA);
        *abort_v = 1;
      }
      return;
    }
    if (*abort_v) return;
    const int64_t base = lo + tile * 32;
    const int nrows = (int)(hi - base < 32 ? hi - base : 32);
    warp_copy_rows_w<W, SplitTuning<KT>::kLoads>(src_s[s], out + base * (int64_t)row_bytes,
                                                 nrows, row_bytes, width, lane);
    __syncwarp();
    if (lane == 0) mbar_arrive(saddr(&empty_bar[s]));
  }
}

using SplitFn = void (*)(TableView, const int32_t*, int64_t, int32_t, uint8_t*, int32_t*,
                         uint8_t*, int, int);

template <int W>
SplitFn pick_split_w(int fmt, int K) {
  if (fmt == FMT16) {
    if (K <= 3) return embed_split_kernel<FMT16, 3, W>;
    if (K <= 5) return embed_split_kernel<FMT16, 5, W>;
    return embed_split_kernel<FMT16, 8, W>;
  }
  if (K <= 5) return embed_split_kernel<FMT32, 5, W>;
  return embed_split_kernel<FMT32, 8, W>;
}

int split_match_warps(int K) {
  if (K <= 3) return SplitTuning<3>::kMatchWarps;
  if (K <= 5) return SplitTuning<5>::kMatchWarps;
  return SplitTuning<8>::kMatchWarps;
}

}  // namespace

int launch_embed_split(const scone_table* tb, const int32_t* tok, int64_t n, int32_t L,
                       uint8_t* out, int32_t* row, uint8_t* len, cudaStream_t stream) {
  const int width = row_copy_width(tb->view, out);
  const SplitFn fn = width == 16 ? pick_split_w<16>(tb->fmt, tb->view.K)
                                 : pick_split_w<0>(tb->fmt, tb->view.K);
  const int n_match = split_match_warps(tb->view.K);
  // every resident block, unless a block would get less than one tile per warp
  const int64_t cap = (int64_t)sm_count() * blocks_per_sm((const void*)fn, kSplitThreads, 0);
  const int64_t need = (n + 32 * kSplitWarps - 1) / (32 * kSplitWarps);
  const int grid = (int)(need < cap ? (need < 1 ? 1 : need) : cap);
  fn<<<grid, kSplitThreads, 0, stream>>>(tb->view, tok, n, L, out, row, len, width, n_match);
  return cudaGetLastError() == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}

}  // namespace scone
