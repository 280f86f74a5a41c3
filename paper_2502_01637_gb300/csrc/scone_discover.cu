// f-gram discovery (C ABI): Algorithm 3 ("Constructing a set of f-grams",
// Appendix A) computed by the K-1 counting scans of Sec. 3.2.
//
// Scan n (n = 2..K) counts the n-grams of the corpus in a GPU hash table.
// An n-gram is keyed by the pair (name of its (n-1)-prefix, last token), where
// the name of an eligible (n-1)-gram is the start of its first occurrence,
// found by the previous scan, and the name of a token is the token itself.
// So every key is one 64-bit word at every length, and no scan re-reads the
// n tokens of a window. A window is counted only when its (n-1)-prefix and its
// (n-1)-suffix are both frequent (count >= min_count): an n-gram that reaches
// min_count has a prefix and a suffix that appear at least as often, so the
// pruning drops no frequent n-gram (Sec. 3.2).
//
// Per scan, over the flattened B x L corpus (positions i, window ending at i):
//   1. count_kernel: every window adds itself to the global table {key,
//      count, ~first} with atomics, except windows whose key sits in their
//      block's shared-memory cache of hot keys, which are counted there and
//      flushed once at the end. Hot keys of a Zipf corpus therefore cost one
//      global update per block, not one per occurrence. Each position keeps
//      the global slot of its window.
//   2. flag_kernel: a window is the first occurrence of a frequent n-gram
//      when its start equals its slot's first occurrence and the count
//      reaches min_count; one bit per position, counted per 1024 positions.
//      Each position also takes the name of its window's n-gram (or none):
//      the prefix and suffix names of the next scan.
//   3. scan_kernel: exclusive prefix sum of those counts.
//   4. assign_kernel: flagged positions, in position order, get consecutive
//      ids; each writes its n-gram's tokens and count to the list of length
//      n. The ids of length n are thus ranks in first-occurrence order.
//
// Selection: the frequent n-grams of all lengths, concatenated by length and
// then first occurrence, are ranked by count, ties by length then first
// occurrence (the reading of "breaking ties arbitrarily" that makes the result
// unique). The S-th largest count c* is found by a radix select on the 32-bit
// counts (four histogram passes of 8 bits); every n-gram above c* is taken,
// and of those equal to c* the first S - #(count > c*) in list order. One
// ordered pass emits the selection, padded to K tokens, in list order.

#include <chrono>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

#include "scone_device.cuh"
#include "scone_host.h"

namespace scone {

namespace {

constexpr uint32_t kNone = 0xFFFFFFFFu;
// Counting kernel shape. Measured on the 1.07e9-token workload, 256..1024
// threads and 1024..2048 cache slots, and tables of load factor 0.1..0.5, all
// ran within 3%: the kernel is bound by the random global updates.
constexpr int kCountThreads = 512;
constexpr int kHotSlots = 2048;                 // per-block cache of hot keys (power of 2)
constexpr int kWin = 4;                         // windows in flight per thread
constexpr uint32_t kHotTag = 0x80000000u;       // slot_of tag: a cache slot, not a table slot
constexpr int kWarpSpan = 1024;           // positions (or list entries) per warp chunk
constexpr int kScanThreads = 1024;
constexpr uint64_t kDiscoverSeed = 0xBB67AE8584CAA73Bull;  // frac(sqrt 3), first 64 bits

// Global counting slot: one 16-byte slot, so a key's count and first
// occurrence share its 32-byte sector. first_inv holds ~start: atomicMax of
// the complement keeps the smallest start, and a zeroed slot is empty.
struct alignas(16) CountSlot {
  unsigned long long key;   // 0 = empty
  unsigned int count;
  unsigned int first_inv;
};

struct DiscoverErr {
  int token_range;
  int table_full;
};

__device__ __forceinline__ uint64_t slot_home(uint64_t key, uint64_t cap) {
  return __umul64hi(fmix64(key ^ kDiscoverSeed), cap);  // fastrange (Lemire 2019)
}

__device__ __forceinline__ uint32_t lanemask_lt() {
  uint32_t m;
  asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
  return m;
}

// Finishes the linear probe of key whose CAS at slot s returned prev: a
// probe is one CAS of the empty key, which either claims the slot or returns
// the key already there.
__device__ __forceinline__ uint32_t probe_rest(CountSlot* table, uint64_t cap, uint64_t key,
                                               uint64_t s, unsigned long long prev,
                                               DiscoverErr* err) {
  for (uint64_t probe = 1; probe < cap; ++probe) {
    if (prev == 0 || prev == key) return (uint32_t)s;
    s = s + 1 == cap ? 0 : s + 1;
    prev = atomicCAS(&table[s].key, 0ull, (unsigned long long)key);
  }
  if (prev == 0 || prev == key) return (uint32_t)s;
  atomicExch(&err->table_full, 1);
  return kNone;
}

// Step 1. names == nullptr for n = 2 (the prefix name is the previous token).
// One thread per window (grid-stride over a persistent grid). A block keeps a
// direct-mapped cache of kHotSlots keys in shared memory for its whole run:
// a window whose key holds (or claims) its cache slot is counted there with
// shared-memory atomics; any other window goes straight to the global table
// (CAS probe, then count and first occurrence as fire-and-forget
// reductions). Frequent keys take their cache slots early, so the hot keys of
// a Zipf corpus reach the global table once per block instead of once per
// occurrence, and no window waits on a barrier. At the end the block flushes
// its cache and rewrites the cached windows' slots (tagged kHotTag) to global.
__global__ void __launch_bounds__(kCountThreads)
count_kernel(const int32_t* __restrict__ tok, const uint32_t* __restrict__ names, int64_t N,
             int32_t L, int32_t n, int32_t vocab, CountSlot* __restrict__ table, uint64_t cap,
             uint32_t* __restrict__ slot_of, unsigned long long* __restrict__ n_cand,
             unsigned long long* __restrict__ n_flush, DiscoverErr* err) {
  __shared__ unsigned long long hkey[kHotSlots];
  __shared__ uint32_t hcnt[kHotSlots];
  __shared__ uint32_t hfirst[kHotSlots];
  __shared__ uint32_t hglob[kHotSlots];
  for (int h = threadIdx.x; h < kHotSlots; h += kCountThreads) {
    hkey[h] = 0;
    hcnt[h] = 0;
    hfirst[h] = kNone;
  }
  __syncthreads();

  unsigned long long my_cand = 0, my_flush = 0;
  const int64_t stride = (int64_t)gridDim.x * kCountThreads;
  const int64_t i0 = (int64_t)blockIdx.x * kCountThreads + threadIdx.x;
  // kWin windows per thread and pass (i, i + stride, ...), so that their
  // loads and their global CAS operations are in flight together
  for (int64_t ib = i0; ib < N; ib += stride * kWin) {
    uint64_t key[kWin];
    uint32_t start[kWin], out[kWin];
    bool cold[kWin];
#pragma unroll
    for (int u = 0; u < kWin; ++u) {
      const int64_t i = ib + u * stride;
      key[u] = 0;
      out[u] = kNone;
      cold[u] = false;
      start[u] = 0;
      if (i >= N) continue;
      const int32_t t = tok[i];
      bool cand = true;
      uint32_t pre = 0;
      if (n == 2 && (t < 0 || t >= vocab)) {
        atomicExch(&err->token_range, 1);
        cand = false;
      }
      if (cand && i % L < n - 1) cand = false;
      if (cand) {
        if (n == 2) {
          const int32_t tp = tok[i - 1];
          cand = tp >= 0 && tp < vocab;
          pre = (uint32_t)tp;
        } else {
          pre = names[i - 1];
          cand = pre != kNone && names[i] != kNone;
        }
      }
      if (cand) {
        key[u] = ((uint64_t)(pre + 1u) << 32) | (uint32_t)t;
        start[u] = (uint32_t)(i - n + 1);
      }
    }
    // the block's cache first; the windows it does not take go global
    uint64_t home[kWin];
    unsigned long long prev[kWin];
#pragma unroll
    for (int u = 0; u < kWin; ++u) {
      if (!key[u]) continue;
      ++my_cand;
      const uint32_t h = (uint32_t)(fmix64(key[u]) & (kHotSlots - 1));
      const unsigned long long hp = atomicCAS(&hkey[h], 0ull, (unsigned long long)key[u]);
      if (hp == 0 || hp == key[u]) {
        atomicAdd(&hcnt[h], 1u);
        atomicMin(&hfirst[h], start[u]);
        out[u] = kHotTag | h;
      } else {
        cold[u] = true;
        home[u] = slot_home(key[u], cap);
        prev[u] = atomicCAS(&table[home[u]].key, 0ull, (unsigned long long)key[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < kWin; ++u) {
      if (cold[u]) {
        const uint32_t g = probe_rest(table, cap, key[u], home[u], prev[u], err);
        ++my_flush;
        if (g != kNone) {
          atomicAdd(&table[g].count, 1u);
          atomicMax(&table[g].first_inv, ~start[u]);
        }
        out[u] = g;
      }
      const int64_t i = ib + u * stride;
      if (i < N) slot_of[i] = out[u];
    }
  }
  __syncthreads();
  // flush the cache: the first probe of every owned slot is issued before
  // any result is used
  constexpr int kOwn = kHotSlots / kCountThreads;
  constexpr int kFlushBatch = kOwn < 4 ? kOwn : 4;
  static_assert(kHotSlots % kCountThreads == 0 && kOwn % kFlushBatch == 0,
                "every cache slot must be owned by exactly one thread");
#pragma unroll
  for (int h0 = 0; h0 < kOwn; h0 += kFlushBatch) {
    unsigned long long key[kFlushBatch], prev[kFlushBatch];
    uint64_t home[kFlushBatch];
#pragma unroll
    for (int k = 0; k < kFlushBatch; ++k) {
      key[k] = hkey[threadIdx.x + (h0 + k) * kCountThreads];
      home[k] = key[k] ? slot_home(key[k], cap) : 0;
      prev[k] = key[k] ? atomicCAS(&table[home[k]].key, 0ull, key[k]) : 0ull;
    }
#pragma unroll
    for (int k = 0; k < kFlushBatch; ++k) {
      const int h = threadIdx.x + (h0 + k) * kCountThreads;
      hglob[h] = kNone;
      if (!key[k]) continue;
      const uint32_t g = probe_rest(table, cap, key[k], home[k], prev[k], err);
      hglob[h] = g;
      ++my_flush;
      if (g == kNone) continue;
      atomicAdd(&table[g].count, hcnt[h]);
      atomicMax(&table[g].first_inv, ~hfirst[h]);
    }
  }
  __syncthreads();
  for (int64_t i = i0; i < N; i += stride) {
    const uint32_t v = slot_of[i];
    if (v != kNone && (v & kHotTag)) slot_of[i] = hglob[v & (kHotSlots - 1)];
  }
  for (int o = 16; o > 0; o >>= 1) {
    my_cand += __shfl_down_sync(0xFFFFFFFFu, my_cand, o);
    my_flush += __shfl_down_sync(0xFFFFFFFFu, my_flush, o);
  }
  if ((threadIdx.x & 31) == 0 && my_cand) atomicAdd(n_cand, my_cand);
  if ((threadIdx.x & 31) == 0 && my_flush) atomicAdd(n_flush, my_flush);
}

// Step 2. One warp per 1024 positions; lane = position within 32.
__global__ void __launch_bounds__(256)
flag_kernel(const uint32_t* __restrict__ slot_of, const CountSlot* __restrict__ table, int64_t N,
            int32_t n, uint32_t min_count, uint32_t* __restrict__ flags,
            uint32_t* __restrict__ chunk_cnt, uint32_t* __restrict__ name_out,
            unsigned long long* __restrict__ n_distinct,
            unsigned long long* __restrict__ n_named) {
  const int lane = threadIdx.x & 31;
  const int64_t n_wchunks = (N + kWarpSpan - 1) / kWarpSpan;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  unsigned long long distinct = 0, named = 0;
  for (int64_t wc = blockIdx.x * (int64_t)(blockDim.x / 32) + threadIdx.x / 32; wc < n_wchunks;
       wc += warps) {
    uint32_t cnt = 0;
    // batches of kBatch positions per lane: all their slot reads in flight at once
    constexpr int kBatch = 8;
    for (int it0 = 0; it0 < kWarpSpan / 32; it0 += kBatch) {
      uint32_t sl[kBatch];
      uint2 cf[kBatch];
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        const int64_t i = wc * kWarpSpan + (it0 + b) * 32 + lane;
        sl[b] = i < N ? slot_of[i] : kNone;
      }
#pragma unroll
      for (int b = 0; b < kBatch; ++b)
        cf[b] = sl[b] != kNone ? *reinterpret_cast<const uint2*>(&table[sl[b]].count)
                               : make_uint2(0u, 0u);
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        const int64_t i = wc * kWarpSpan + (it0 + b) * 32 + lane;
        const bool first = sl[b] != kNone && ~cf[b].y == (uint32_t)(i - n + 1);
        const bool freq = first && cf[b].x >= min_count;
        if (name_out && i < N) {
          // name of the window's n-gram for the next scan: its first occurrence
          const bool eligible = sl[b] != kNone && cf[b].x >= min_count;
          name_out[i] = eligible ? ~cf[b].y : kNone;
          named += eligible;
        }
        const uint32_t word = __ballot_sync(0xFFFFFFFFu, freq);
        const uint32_t dword = __ballot_sync(0xFFFFFFFFu, first);
        if (lane == 0 && wc * kWarpSpan + (it0 + b) * 32 < N)
          flags[(wc * kWarpSpan) / 32 + it0 + b] = word;
        cnt += __popc(word);
        distinct += __popc(dword);
      }
    }
    if (lane == 0) chunk_cnt[wc] = cnt;
  }
  if (lane == 0 && distinct) atomicAdd(n_distinct, distinct);
  for (int o = 16; o > 0; o >>= 1) named += __shfl_down_sync(0xFFFFFFFFu, named, o);
  if (lane == 0 && named) atomicAdd(n_named, named);
}

// Step 3 (and the selection's offsets): exclusive prefix sum of n counts by
// one block; total receives the sum.
__global__ void __launch_bounds__(kScanThreads)
scan_kernel(const uint32_t* __restrict__ in, unsigned long long* __restrict__ out, int64_t n,
            unsigned long long* __restrict__ total) {
  __shared__ unsigned long long warp_sums[kScanThreads / 32];
  const int64_t per = (n + kScanThreads - 1) / kScanThreads;
  const int64_t b = threadIdx.x * per;
  const int64_t e = b + per < n ? b + per : n;
  unsigned long long sum = 0;
  for (int64_t k = b; k < e; ++k) sum += in[k];
  // block exclusive scan of the per-thread sums
  const int lane = threadIdx.x & 31, warp = threadIdx.x / 32;
  unsigned long long incl = sum;
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) warp_sums[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    unsigned long long w = warp_sums[lane];
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long v = __shfl_up_sync(0xFFFFFFFFu, w, o);
      if (lane >= o) w += v;
    }
    warp_sums[lane] = w;   // inclusive over warps
  }
  __syncthreads();
  unsigned long long run = incl - sum + (warp > 0 ? warp_sums[warp - 1] : 0ull);
  for (int64_t k = b; k < e; ++k) {
    out[k] = run;
    run += in[k];
  }
  if (threadIdx.x == kScanThreads - 1) *total = warp_sums[31];
}

// Step 4. One warp per 1024 positions, in position order.
__global__ void __launch_bounds__(256)
assign_kernel(const uint32_t* __restrict__ flags, const unsigned long long* __restrict__ chunk_off,
              const uint32_t* __restrict__ slot_of, const CountSlot* __restrict__ table,
              const int32_t* __restrict__ tok, int64_t N, int32_t n,
              int32_t* __restrict__ list_tok, uint32_t* __restrict__ list_cnt) {
  const int lane = threadIdx.x & 31;
  const int64_t n_wchunks = (N + kWarpSpan - 1) / kWarpSpan;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t wc = blockIdx.x * (int64_t)(blockDim.x / 32) + threadIdx.x / 32; wc < n_wchunks;
       wc += warps) {
    const int64_t w0 = (wc * kWarpSpan) / 32;
    const int64_t n_words = (N + 31) / 32;
    const uint32_t my_word = w0 + lane < n_words ? flags[w0 + lane] : 0u;
    unsigned long long off = chunk_off[wc];
    for (int it = 0; it < kWarpSpan / 32; ++it) {
      const uint32_t word = __shfl_sync(0xFFFFFFFFu, my_word, it);
      if (word == 0) continue;
      if ((word >> lane) & 1u) {
        const int64_t i = wc * kWarpSpan + it * 32 + lane;
        const uint64_t id = off + __popc(word & lanemask_lt());
        const uint32_t sl = slot_of[i];
        list_cnt[id] = table[sl].count;
        for (int j = 0; j < n; ++j) list_tok[id * n + j] = tok[i - n + 1 + j];
      }
      off += __popc(word);
    }
  }
}

// The per-length lists seen as one concatenated list (length ascending).
struct Lists {
  const uint32_t* cnt[8];
  const int32_t* tok[8];
  int64_t size[8];
  int64_t chunk_base[8];   // first warp chunk of each list in the concatenated chunk array
  int32_t len[8];
  int32_t n_lists;
};

// Radix-select pass: histogram of byte (c >> shift) & 255 over the counts c
// with (c & mask) == prefix. grid.y = list.
__global__ void __launch_bounds__(256)
hist_kernel(Lists ls, int shift, uint32_t mask, uint32_t prefix, unsigned int* __restrict__ hist) {
  __shared__ unsigned int h[256];
  h[threadIdx.x] = 0;
  __syncthreads();
  const int q = blockIdx.y;
  const uint32_t* cnt = ls.cnt[q];
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < ls.size[q];
       e += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t c = cnt[e];
    if ((c & mask) == prefix) atomicAdd(&h[(c >> shift) & 255u], 1u);
  }
  __syncthreads();
  if (h[threadIdx.x]) atomicAdd(&hist[threadIdx.x], h[threadIdx.x]);
}

// Per warp chunk of a list: how many counts are above c* and how many equal.
__global__ void __launch_bounds__(256)
select_count_kernel(Lists ls, uint32_t cstar, uint32_t* __restrict__ chunk_gt,
                    uint32_t* __restrict__ chunk_eq) {
  const int lane = threadIdx.x & 31;
  const int q = blockIdx.y;
  const int64_t size = ls.size[q];
  const int64_t n_wchunks = (size + kWarpSpan - 1) / kWarpSpan;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t wc = blockIdx.x * (int64_t)(blockDim.x / 32) + threadIdx.x / 32; wc < n_wchunks;
       wc += warps) {
    uint32_t gt = 0, eq = 0;
    for (int it = 0; it < kWarpSpan / 32; ++it) {
      const int64_t e = wc * kWarpSpan + it * 32 + lane;
      const uint32_t c = e < size ? ls.cnt[q][e] : 0u;
      gt += __popc(__ballot_sync(0xFFFFFFFFu, e < size && c > cstar));
      eq += __popc(__ballot_sync(0xFFFFFFFFu, e < size && c == cstar));
    }
    if (lane == 0) {
      chunk_gt[ls.chunk_base[q] + wc] = gt;
      chunk_eq[ls.chunk_base[q] + wc] = eq;
    }
  }
}

// Emits the selection in list order: entry e goes to #(count > c* before e)
// + min(#(count == c* before e), take_eq) when it is selected.
__global__ void __launch_bounds__(256)
emit_kernel(Lists ls, uint32_t cstar, unsigned long long take_eq,
            const unsigned long long* __restrict__ gt_off,
            const unsigned long long* __restrict__ eq_off, int32_t K,
            int32_t* __restrict__ out_tok, uint8_t* __restrict__ out_len,
            uint32_t* __restrict__ out_cnt) {
  const int lane = threadIdx.x & 31;
  const int q = blockIdx.y;
  const int64_t size = ls.size[q];
  const int n = ls.len[q];
  const int64_t n_wchunks = (size + kWarpSpan - 1) / kWarpSpan;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x / 32);
  for (int64_t wc = blockIdx.x * (int64_t)(blockDim.x / 32) + threadIdx.x / 32; wc < n_wchunks;
       wc += warps) {
    unsigned long long g = gt_off[ls.chunk_base[q] + wc];
    unsigned long long qe = eq_off[ls.chunk_base[q] + wc];
    for (int it = 0; it < kWarpSpan / 32; ++it) {
      const int64_t e = wc * kWarpSpan + it * 32 + lane;
      const uint32_t c = e < size ? ls.cnt[q][e] : 0u;
      const bool gt = e < size && c > cstar;
      const bool eq = e < size && c == cstar;
      const uint32_t gm = __ballot_sync(0xFFFFFFFFu, gt);
      const uint32_t em = __ballot_sync(0xFFFFFFFFu, eq);
      const unsigned long long my_g = g + __popc(gm & lanemask_lt());
      const unsigned long long my_e = qe + __popc(em & lanemask_lt());
      if (gt || (eq && my_e < take_eq)) {
        const unsigned long long o = my_g + (my_e < take_eq ? my_e : take_eq);
        const int32_t* src = ls.tok[q] + e * n;
        for (int j = 0; j < K; ++j) out_tok[o * K + j] = j < n ? src[j] : -1;
        out_len[o] = (uint8_t)n;
        if (out_cnt) out_cnt[o] = c;
      }
      g += __popc(gm);
      qe += __popc(em);
    }
  }
}

// CUDA events of one call (timing for the statistics), destroyed on exit.
struct Events {
  std::vector<cudaEvent_t> ev;
  cudaEvent_t make() {
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    ev.push_back(e);
    return e;
  }
  ~Events() {
    for (cudaEvent_t e : ev) cudaEventDestroy(e);
  }
};

double elapsed_ms(cudaEvent_t a, cudaEvent_t b) {
  float ms = 0.f;
  if (!a || !b || cudaEventElapsedTime(&ms, a, b) != cudaSuccess) {
    cudaGetLastError();
    return 0.0;
  }
  return ms;
}

// Named buffers of a workspace.
enum Buf {
  kBufNames, kBufSlotOf, kBufFlags, kBufChunkCnt, kBufChunkOff, kBufCounters, kBufErr, kBufTable,
  kBufHist, kBufGt, kBufEq, kBufGtOff, kBufEqOff,
  kBufListCnt,                 // + n, n = 0..8
  kBufListTok = kBufListCnt + 9,
  kBufCount = kBufListTok + 9
};

}  // namespace
}  // namespace scone

// Reusable device workspace: grow-only buffers, kept between calls.
struct scone_discover {
  int device = 0;
  void* ptr[scone::kBufCount] = {};
  size_t bytes[scone::kBufCount] = {};
  double host_ms = 0.0;      // host time spent in allocation calls of the current call

  void* get(int b, size_t need) {
    if (need == 0) need = 16;
    if (bytes[b] >= need) return ptr[b];
    const auto t0 = std::chrono::steady_clock::now();
    if (ptr[b]) cudaFree(ptr[b]);
    ptr[b] = nullptr;
    bytes[b] = 0;
    const size_t want = ((need + need / 8) + ((size_t)1 << 21) - 1) & ~(((size_t)1 << 21) - 1);
    void* p = nullptr;
    const cudaError_t rc = cudaMalloc(&p, want);
    host_ms += std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0)
                   .count();
    if (rc != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
    ptr[b] = p;
    bytes[b] = want;
    return p;
  }
  size_t total() const {
    size_t t = 0;
    for (size_t b : bytes) t += b;
    return t;
  }
  ~scone_discover() {
    for (void* p : ptr)
      if (p) cudaFree(p);
  }
};

namespace scone {
namespace {

int grid_for(const void* fn, int threads, size_t smem, int64_t work_blocks) {
  const int64_t resident = (int64_t)blocks_per_sm(fn, threads, smem) * sm_count();
  int64_t g = work_blocks < resident ? work_blocks : resident;
  return (int)(g < 1 ? 1 : g);
}

}  // namespace

}  // namespace scone

using namespace scone;

extern "C" int scone_discover_create(scone_discover** out) {
  if (!out) return SCONE_ERR_INVALID_ARG;
  *out = nullptr;
  auto* ws = new (std::nothrow) scone_discover();
  if (!ws) return SCONE_ERR_NOMEM;
  if (cudaGetDevice(&ws->device) != cudaSuccess) {
    cudaGetLastError();
    delete ws;
    return SCONE_ERR_CUDA;
  }
  *out = ws;
  return SCONE_OK;
}

extern "C" int scone_discover_destroy(scone_discover* ws) {
  if (!ws) return SCONE_OK;
  DeviceGuard dg(ws->device);
  delete ws;
  return SCONE_OK;
}

extern "C" int scone_fgram_discover(scone_discover* ws, const int32_t* tok, int32_t B, int32_t L, int32_t vocab,
                                    int32_t K, int64_t S, int32_t min_count, int32_t* fgram_tok,
                                    uint8_t* fgram_len, uint32_t* fgram_count, int64_t* n_out,
                                    scone_discover_stats* stats, void* stream) {
  if (B < 0 || L < 0 || vocab < 1 || K < 2 || K > 8 || S < 0 || min_count < 1 || !n_out)
    return SCONE_ERR_INVALID_ARG;
  const int64_t N = (int64_t)B * L;
  if (N > (1ll << 30)) return SCONE_ERR_UNSUPPORTED;   // table slots must stay below kHotTag
  if (N > 0 && !tok) return SCONE_ERR_INVALID_ARG;
  if (S > 0 && (!fgram_tok || !fgram_len)) return SCONE_ERR_INVALID_ARG;
  *n_out = 0;
  scone_discover_stats st;
  std::memset(&st, 0, sizeof(st));
  if (stats) *stats = st;
  if (N == 0) return SCONE_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);


  Events evs;
  cudaEvent_t ev_begin = evs.make(), ev_end = evs.make();
  cudaEvent_t ev_c0[9], ev_c1[9], ev_s0[9], ev_s1[9];
  for (int n = 0; n <= 8; ++n) {
    ev_c0[n] = evs.make();
    ev_c1[n] = evs.make();
    ev_s0[n] = evs.make();
    ev_s1[n] = evs.make();
  }
  cudaEvent_t ev_sel = evs.make();
  if (ev_begin) cudaEventRecord(ev_begin, s);

  // the caller's workspace, or one for this call only
  scone_discover* tmp = nullptr;
  if (!ws) {
    tmp = new (std::nothrow) scone_discover();
    if (!tmp) return SCONE_ERR_NOMEM;
    cudaGetDevice(&tmp->device);
    ws = tmp;
  }
  struct TmpGuard {
    scone_discover* p;
    ~TmpGuard() { delete p; }
  } tmp_guard{tmp};
  DeviceGuard dg(ws->device);
  ws->host_ms = 0.0;
  bool nomem = false;
  auto get = [&](int b, size_t need) -> void* {
    void* p = ws->get(b, need);
    if (!p) nomem = true;
    return p;
  };
  const int64_t n_words = (N + 31) / 32;
  const int64_t n_wchunks = (N + kWarpSpan - 1) / kWarpSpan;
  auto* names = static_cast<uint32_t*>(get(kBufNames, (size_t)N * 4));
  auto* slot_of = static_cast<uint32_t*>(get(kBufSlotOf, (size_t)N * 4));
  auto* flags = static_cast<uint32_t*>(get(kBufFlags, (size_t)n_words * 4));
  auto* chunk_cnt = static_cast<uint32_t*>(get(kBufChunkCnt, (size_t)n_wchunks * 4));
  auto* chunk_off = static_cast<unsigned long long*>(get(kBufChunkOff, (size_t)n_wchunks * 8));
  auto* counters = static_cast<unsigned long long*>(get(kBufCounters, 8 * 8));
  auto* d_err = static_cast<DiscoverErr*>(get(kBufErr, sizeof(DiscoverErr)));
  if (nomem) return SCONE_ERR_NOMEM;
  if (cudaMemsetAsync(d_err, 0, sizeof(DiscoverErr), s) != cudaSuccess) return SCONE_ERR_CUDA;

  std::vector<uint32_t*> list_cnt(K + 1, nullptr);
  std::vector<int32_t*> list_tok(K + 1, nullptr);
  std::vector<int64_t> list_size(K + 1, 0);

  int64_t cand_bound = (int64_t)B * (L > 0 ? L - 1 : 0);   // windows of length 2
  for (int n = 2; n <= K; ++n) {
    if (cand_bound == 0 && n > 2) break;   // scan 2 always runs: it checks every token
    if (ev_s0[n]) cudaEventRecord(ev_s0[n], s);
    // at most one distinct n-gram per counted window: load factor <= 0.5
    const uint64_t cap = (uint64_t)(2 * cand_bound > 64 ? 2 * cand_bound : 64);
    auto* table = static_cast<CountSlot*>(get(kBufTable, (size_t)cap * sizeof(CountSlot)));
    if (nomem) return SCONE_ERR_NOMEM;
    if (cudaMemsetAsync(table, 0, cap * sizeof(CountSlot), s) != cudaSuccess ||
        cudaMemsetAsync(counters, 0, 8 * sizeof(unsigned long long), s) != cudaSuccess)
      return SCONE_ERR_CUDA;

    if (ev_c0[n]) cudaEventRecord(ev_c0[n], s);
    count_kernel<<<grid_for((const void*)count_kernel, kCountThreads, 0,
                            (N + kCountThreads - 1) / kCountThreads),
                   kCountThreads, 0, s>>>(tok, n == 2 ? nullptr : names, N, L, n, vocab,
                                                   table, cap, slot_of, counters + 0,
                                                   counters + 6, d_err);
    if (ev_c1[n]) cudaEventRecord(ev_c1[n], s);
    const int gw = grid_for((const void*)flag_kernel, 256, 0, (n_wchunks + 7) / 8);
    flag_kernel<<<gw, 256, 0, s>>>(slot_of, table, N, n, (uint32_t)min_count, flags, chunk_cnt,
                                   n < K ? names : nullptr, counters + 1, counters + 3);
    scan_kernel<<<1, kScanThreads, 0, s>>>(chunk_cnt, chunk_off, n_wchunks, counters + 2);
    if (cudaGetLastError() != cudaSuccess) return SCONE_ERR_CUDA;
    unsigned long long h[7];
    DiscoverErr herr;
    if (cudaMemcpyAsync(h, counters, sizeof(h), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaMemcpyAsync(&herr, d_err, sizeof(herr), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
      return SCONE_ERR_CUDA;
    if (herr.token_range) return SCONE_ERR_TOKEN_RANGE;
    if (herr.table_full) return SCONE_ERR_TABLE_FULL;
    st.candidates[n] = (int64_t)h[0];
    st.distinct[n] = (int64_t)h[1];
    st.frequent[n] = (int64_t)h[2];
    st.flushes[n] = (int64_t)h[6];
    st.ms_count[n] = elapsed_ms(ev_c0[n], ev_c1[n]);
    const int64_t M = (int64_t)h[2];
    list_size[n] = M;
    list_cnt[n] = static_cast<uint32_t*>(get(kBufListCnt + n, (size_t)M * 4));
    list_tok[n] = static_cast<int32_t*>(get(kBufListTok + n, (size_t)M * n * 4));
    if (nomem) return SCONE_ERR_NOMEM;
    if (M > 0)
      assign_kernel<<<gw, 256, 0, s>>>(flags, chunk_off, slot_of, table, tok, N, n,
                                       list_tok[n], list_cnt[n]);
    // windows of eligible n-grams bound the windows of the next scan
    cand_bound = n < K && M > 0 ? (int64_t)h[3] : 0;
    if (cudaGetLastError() != cudaSuccess) return SCONE_ERR_CUDA;
    st.table_bytes_max = st.table_bytes_max > (int64_t)(cap * sizeof(CountSlot))
                             ? st.table_bytes_max
                             : (int64_t)(cap * sizeof(CountSlot));
    if (ev_s1[n] && cudaEventRecord(ev_s1[n], s) == cudaSuccess &&
        cudaEventSynchronize(ev_s1[n]) == cudaSuccess)
      st.ms_scan[n] = elapsed_ms(ev_s0[n], ev_s1[n]);
  }
  if (ev_sel) cudaEventRecord(ev_sel, s);

  // Selection over the concatenated lists.
  Lists ls;
  std::memset(&ls, 0, sizeof(ls));
  int64_t M_total = 0, chunks_total = 0;
  for (int n = 2; n <= K; ++n) {
    if (list_size[n] == 0) continue;
    const int q = ls.n_lists++;
    ls.cnt[q] = list_cnt[n];
    ls.tok[q] = list_tok[n];
    ls.size[q] = list_size[n];
    ls.len[q] = n;
    ls.chunk_base[q] = chunks_total;
    chunks_total += (list_size[n] + kWarpSpan - 1) / kWarpSpan;
    M_total += list_size[n];
  }
  const int64_t n_sel = S < M_total ? S : M_total;
  if (n_sel == 0) {
    if (ev_end && cudaEventRecord(ev_end, s) == cudaSuccess &&
        cudaEventSynchronize(ev_end) == cudaSuccess)
      st.ms_total = elapsed_ms(ev_begin, ev_end);
    st.ms_alloc_host = ws->host_ms;
    st.workspace_bytes = (int64_t)ws->total();
    if (stats) *stats = st;
    return SCONE_OK;
  }
  uint32_t cstar = 0;               // with c* = 0 every entry is above it: all selected
  unsigned long long take_eq = 0;
  if (S < M_total) {
    auto* hist = static_cast<unsigned int*>(get(kBufHist, 256 * 4));
    if (nomem) return SCONE_ERR_NOMEM;
    uint32_t mask = 0, prefix = 0;
    int64_t k = S;                  // rank still to find among entries matching prefix
    int64_t max_size = 0;
    for (int q = 0; q < ls.n_lists; ++q) max_size = ls.size[q] > max_size ? ls.size[q] : max_size;
    const dim3 hg((unsigned)grid_for((const void*)hist_kernel, 256, 0, (max_size + 255) / 256),
                  (unsigned)ls.n_lists);
    for (int shift = 24; shift >= 0; shift -= 8) {
      unsigned int hh[256];
      if (cudaMemsetAsync(hist, 0, 256 * sizeof(unsigned int), s) != cudaSuccess)
        return SCONE_ERR_CUDA;
      hist_kernel<<<hg, 256, 0, s>>>(ls, shift, mask, prefix, hist);
      if (cudaGetLastError() != cudaSuccess ||
          cudaMemcpyAsync(hh, hist, sizeof(hh), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
          cudaStreamSynchronize(s) != cudaSuccess)
        return SCONE_ERR_CUDA;
      int b = 255;
      for (; b > 0; --b) {
        if ((int64_t)hh[b] >= k) break;
        k -= hh[b];
      }
      prefix |= (uint32_t)b << shift;
      mask |= 255u << shift;
    }
    cstar = prefix;
    take_eq = (unsigned long long)k;
  }
  st.threshold = (int64_t)cstar;
  st.selected_at_threshold = (int64_t)take_eq;

  auto* c_gt = static_cast<uint32_t*>(get(kBufGt, (size_t)chunks_total * 4));
  auto* c_eq = static_cast<uint32_t*>(get(kBufEq, (size_t)chunks_total * 4));
  auto* o_gt = static_cast<unsigned long long*>(get(kBufGtOff, (size_t)chunks_total * 8));
  auto* o_eq = static_cast<unsigned long long*>(get(kBufEqOff, (size_t)chunks_total * 8));
  if (nomem) return SCONE_ERR_NOMEM;
  int64_t max_chunks = 0;
  for (int q = 0; q < ls.n_lists; ++q) {
    const int64_t c = (ls.size[q] + kWarpSpan - 1) / kWarpSpan;
    max_chunks = c > max_chunks ? c : max_chunks;
  }
  const dim3 sg((unsigned)grid_for((const void*)select_count_kernel, 256, 0, (max_chunks + 7) / 8),
                (unsigned)ls.n_lists);
  select_count_kernel<<<sg, 256, 0, s>>>(ls, cstar, c_gt, c_eq);
  scan_kernel<<<1, kScanThreads, 0, s>>>(c_gt, o_gt, chunks_total, counters + 4);
  scan_kernel<<<1, kScanThreads, 0, s>>>(c_eq, o_eq, chunks_total, counters + 5);
  emit_kernel<<<sg, 256, 0, s>>>(ls, cstar, take_eq, o_gt, o_eq, K, fgram_tok, fgram_len,
                                 fgram_count);
  if (ev_end) cudaEventRecord(ev_end, s);
  if (cudaGetLastError() != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess)
    return SCONE_ERR_CUDA;
  st.ms_total = elapsed_ms(ev_begin, ev_end);
  st.ms_select = elapsed_ms(ev_sel, ev_end);
  st.ms_alloc_host = ws->host_ms;
  st.workspace_bytes = (int64_t)ws->total();
  *n_out = n_sel;
  if (stats) *stats = st;
  return SCONE_OK;
}
