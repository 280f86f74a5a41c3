// Fused embed with bulk (TMA) row copies, for large rows in HBM.
//
// Same selection as embed_kernel (Algorithm 1, inference branch, Sec. 3);
// the difference is how rows move. Each CTA owns an even share of the
// positions and runs two roles:
//   * 4 matcher warps: one lane per position, a tile of 128 positions at a
//     time, write the selected row addresses into a double-buffered table
//     in shared memory;
//   * 1 mover warp, whose lane 0 streams the rows through a ring of R
//     row-sized shared-memory slots: cp.async.bulk global -> shared with an
//     mbarrier per slot (completion by transaction bytes), then
//     cp.async.bulk shared -> global into the contiguous output. Stores are
//     committed in groups of G rows; a slot is reloaded once the store group
//     that read it has finished reading (wait_group.read), so up to R - 2G
//     loads stay in flight per CTA without holding any registers.
// Matchers and mover hand over the address tables with named barriers.
// Error positions copy a zero row kept by the table.
//
// Every mbarrier wait is bounded: past kSpinLimit polls the CTA records
// SCONE_ERR_CUDA in the status word, stops issuing copies, keeps taking part
// in the named barriers (so no warp is left waiting) and drains its own
// outstanding bulk operations before returning.

#include "scone_host.h"
#include "scone_ptx.cuh"

namespace scone {

constexpr int kBulkMatchWarps = 4;
constexpr int kBulkThreads = 32 * (1 + kBulkMatchWarps);
constexpr int kBulkTile = 32 * kBulkMatchWarps;
constexpr int kBulkGroup = 4;
constexpr uint32_t kSpinLimit = 1u << 22;

namespace {

__device__ __forceinline__ void bar_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}
__device__ __forceinline__ void bar_arrive(int id, int count) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(count) : "memory");
}


// named barrier ids (0 is __syncthreads)
__device__ __forceinline__ int bar_full(int64_t tile) { return 1 + (int)(tile & 1); }
__device__ __forceinline__ int bar_empty(int64_t tile) { return 3 + (int)(tile & 1); }

template <int FMT, int KT>
__global__ void __launch_bounds__(kBulkThreads)
    embed_bulk_kernel(const TableView t, const int32_t* __restrict__ tok, int64_t n_tok,
                      int32_t L, uint8_t* __restrict__ out, int32_t* __restrict__ row_out,
                      uint8_t* __restrict__ len_out, const uint8_t* __restrict__ zero_row,
                      int ring) {
  extern __shared__ __align__(128) uint8_t smem[];
  const uint32_t row_bytes = (uint32_t)t.d * 2;
  uint8_t* slots = smem;                                                   // [ring][row_bytes]
  const void** srcs = reinterpret_cast<const void**>(smem + (size_t)ring * row_bytes);  // [2][tile]
  uint64_t* full = reinterpret_cast<uint64_t*>(srcs + 2 * kBulkTile);      // [ring]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t lo = n_tok * blockIdx.x / gridDim.x;
  const int64_t hi = n_tok * (blockIdx.x + 1) / gridDim.x;
  const int64_t total = hi - lo;
  const int64_t n_tiles = (total + kBulkTile - 1) / kBulkTile;

  if (threadIdx.x == 0) {
    for (int s = 0; s < ring; ++s) mbar_init(saddr(&full[s]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  if (warp > 0) {
    // ---------------------------------------------------------- matchers
    const int m = threadIdx.x - 32;
    for (int64_t k = 0; k < n_tiles; ++k) {
      if (k >= 2) bar_sync(bar_empty(k), kBulkThreads);
      const int64_t j = k * kBulkTile + m;
      const void* src = zero_row;
      if (j < total) {
        const int64_t p = lo + j;
        const int32_t x = __ldg(tok + p);
        int len = 0, err = 0;
        const int32_t r = match_position<FMT, KT>(t, tok, p, (int32_t)(p % L), x, &len, &err);
        if (err) {
          record_error(t, err);
        } else {
          src = r >= 0 ? static_cast<const void*>(t.F + (int64_t)r * t.d)
                       : static_cast<const void*>(t.T + (int64_t)x * t.d);
        }
        if (row_out) row_out[p] = r;
        if (len_out) len_out[p] = (uint8_t)len;
      }
      srcs[(k & 1) * kBulkTile + m] = src;
      bar_arrive(bar_full(k), kBulkThreads);
    }
    return;
  }

  // ---------------------------------------------------------------- mover
  int64_t ready = 0;      // tiles whose addresses are in shared memory
  int64_t released = 0;   // tiles handed back to the matchers
  int64_t loaded = 0;     // rows handed to issue_load
  int64_t issued = 0;     // lane 0: rows whose bulk loads were really issued
  int64_t waited = 0;     // lane 0: rows whose loads were seen complete
  bool failed = false;

  // all 32 lanes walk the same control flow (named barriers count whole
  // warps); lane 0 issues the copies
  auto issue_load = [&](int64_t j) {
    const int64_t tile = j / kBulkTile;
    while (ready <= tile) {
      bar_sync(bar_full(ready), kBulkThreads);
      ++ready;
    }
    if (lane == 0 && !failed) {
      const int s = (int)(j % ring);
      const uint32_t bar = saddr(&full[s]);
      mbar_expect_tx(bar, row_bytes);
      bulk_load(saddr(slots + (size_t)s * row_bytes),
                srcs[(tile & 1) * kBulkTile + (j % kBulkTile)], row_bytes, bar);
      issued = j + 1;
    }
    // a tile's addresses are no longer needed once its last row is issued;
    // only tiles the matchers will wait for (k + 2 < n_tiles) are released
    const bool tile_done = (j + 1) % kBulkTile == 0 || j + 1 == total;
    if (tile_done) {
      if (released + 2 < n_tiles) bar_arrive(bar_empty(released), kBulkThreads);
      ++released;
    }
  };

  const int64_t prologue = total < ring ? total : ring;
  while (loaded < prologue) issue_load(loaded++);
  for (int64_t g0 = 0; g0 < total; g0 += kBulkGroup) {
    const int64_t g1 = g0 + kBulkGroup < total ? g0 + kBulkGroup : total;
    if (lane == 0) {
      for (int64_t j = g0; j < g1; ++j) {
        const int s = (int)(j % ring);
        const uint32_t parity = (uint32_t)((j / ring) & 1);
        uint32_t spins = 0;
        while (!failed && !mbar_try_wait(saddr(&full[s]), parity)) {
          if (++spins >= kSpinLimit) {
            failed = true;
            record_error(t, SCONE_ERR_CUDA);
          }
        }
        if (!failed) {
          waited = j + 1;
          bulk_store(out + (lo + j) * (int64_t)row_bytes, saddr(slots + (size_t)s * row_bytes),
                     row_bytes);
        }
      }
      bulk_commit();
      // the group before this one has finished reading its slots
      bulk_wait_read_1();
    }
    __syncwarp();
    // refill the slots read by the previous group
    const int64_t limit = g0 + ring < total ? g0 + ring : total;
    while (loaded < limit) issue_load(loaded++);
  }
  if (lane == 0) {
    if (failed) {
      // drain the loads still in flight into the ring before the CTA exits
      for (int64_t j = waited; j < issued; ++j) {
        uint32_t spins = 0;
        while (!mbar_try_wait(saddr(&full[j % ring]), (uint32_t)((j / ring) & 1)) &&
               ++spins < kSpinLimit) {
        }
      }
    }
    bulk_wait_all();
  }
  // tiles whose addresses were never needed (empty CTA tail) still owe the
  // matchers nothing: they only wait on tiles k >= 2 released above
  while (ready < n_tiles) {
    bar_sync(bar_full(ready), kBulkThreads);
    ++ready;
  }
}

using BulkFn = void (*)(TableView, const int32_t*, int64_t, int32_t, uint8_t*, int32_t*, uint8_t*,
                        const uint8_t*, int);

BulkFn pick_bulk(int fmt, int K) {
  if (fmt == FMT16) {
    if (K <= 3) return embed_bulk_kernel<FMT16, 3>;
    if (K <= 5) return embed_bulk_kernel<FMT16, 5>;
    return embed_bulk_kernel<FMT16, 8>;
  }
  if (K <= 5) return embed_bulk_kernel<FMT32, 5>;
  return embed_bulk_kernel<FMT32, 8>;
}

}  // namespace

// Ring slots for a row size: as many as fit in ~200 KB, a multiple of the
// store group, at most 64; 0 when rows are too large for a useful ring.
int bulk_ring_slots(int row_bytes) {
  const int budget = 200 * 1024 - 2 * kBulkTile * 8;
  int r = budget / (row_bytes + 8);
  if (r > 64) r = 64;
  r -= r % kBulkGroup;
  return r >= 3 * kBulkGroup ? r : 0;
}

bool bulk_eligible(const scone_table* tb, const void* out) {
  const TableView& t = tb->view;
  const int row_bytes = t.d * 2;
  if (!tb->zero_row || tb->info.F_location != SCONE_ROWS_DEVICE) return false;
  if (row_bytes % 16 != 0 || bulk_ring_slots(row_bytes) == 0) return false;
  uintptr_t a = (uintptr_t)t.T | (uintptr_t)out;
  if (t.n_fgrams > 0) a |= (uintptr_t)t.F;
  return (a & 15) == 0;
}

int launch_embed_bulk(const scone_table* tb, const int32_t* tok, int64_t n, int32_t L,
                      uint8_t* out, int32_t* row, uint8_t* len, cudaStream_t stream) {
  const TableView& t = tb->view;
  const int row_bytes = t.d * 2;
  const int ring = bulk_ring_slots(row_bytes);
  const size_t smem = (size_t)ring * row_bytes + 2 * kBulkTile * sizeof(void*) + ring * 8;
  const BulkFn fn = pick_bulk(tb->fmt, t.K);
  if (cudaFuncSetAttribute((const void*)fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess) {
    cudaGetLastError();
    return SCONE_ERR_CUDA;
  }
  int64_t grid = sm_count();
  const int64_t want = (n + kBulkTile - 1) / kBulkTile;
  if (want < grid) grid = want < 1 ? 1 : want;
  fn<<<(unsigned)grid, kBulkThreads, smem, stream>>>(t, tok, n, L, out, row, len, tb->zero_row,
                                                     ring);
  return cudaGetLastError() == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}

}  // namespace scone
