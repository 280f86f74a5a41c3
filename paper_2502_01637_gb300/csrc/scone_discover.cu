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
//   1a. bin_kernel: every window's key; windows whose key sits in their
//      block's shared-memory cache of hot keys are counted there (each
//      block's cache goes to a hot list). Every other window becomes a
//      record, grouped per chunk of kChunk windows by the region of the table
//      its key hashes to. Every key also enters a HyperLogLog sketch.
//   The host sizes the counting table {key, count, ~first} from the sketch's
//   estimate of the distinct keys and zeroes it; hotflush_kernel adds the hot
//   lists to it.
//   1b. bincount_kernel: the records, region by region, add themselves to the
//      table with atomics. All blocks work on one or two regions at a time, so
//      the updates hit L2 instead of random DRAM sectors. (If the table fills
//      up, it is rebuilt at the worst-case size and 1b to 2b run again.)
//   2a. flagbin_kernel: the records, region by region again, look their keys
//      up in the finished table (L2 hits). A window is the first occurrence
//      of a frequent n-gram when its start equals the slot's first occurrence
//      and the count reaches min_count; the window's n-gram is named (for the
//      next scan's prefix and suffix) by its first occurrence when frequent.
//   2b. unsort_kernel: per chunk, the records' results back in position
//      order (hot-cached windows look their few keys up directly); one bit
//      per position, counted per 1024 positions, and one name per position.
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
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

#include "scone_device.cuh"
#include "scone_host.h"

namespace scone {

namespace {

constexpr uint32_t kNone = 0xFFFFFFFFu;
// Binning shape. A chunk is kChunk consecutive windows of one binning block;
// its records fall into kBins bins by table region, so a region is cap / 1024
// slots (at most 34 MB at the largest table) and two of them fit in L2.
constexpr int kBinBits = 10;
constexpr int kBins = 1 << kBinBits;
constexpr int kChunk = 16384;                   // windows per chunk (record offsets fit 16 bits)
constexpr int kBinThreads = 1024;
constexpr int kHotSlots = 2048;                 // per-block cache of hot keys (power of 2)
constexpr int kWin = 4;                         // windows (records) in flight per thread
// Counting shape: a block takes kItemChunks chunks of one bin at a time (32
// per warp) and aggregates them in a kCntSlots-slot shared-memory cache. On the
// 1.07e9-token corpus, items of 256 chunks (2,048 slots) counted in 20.4 +
// 20.7 ms per scan, 512 (4,096) in 18.3 + 20.7 and 1,024 (8,192) in 17.0 +
// 21.2; one warp per 32 chunks (256 slots each) in 40 + 34.
constexpr int kCntThreads = 512;
constexpr int kItemChunks = kCntThreads;
constexpr int kCntSlots = 4096;
constexpr size_t kCntSmem = (size_t)kCntSlots * 16;
constexpr int kUnsortThreads = 512;             // 16 warps x 1024 positions = one chunk
// Distinct-key estimate that sizes the counting table: a HyperLogLog sketch
// of 2^12 registers (standard error 1.6%).
constexpr int kHllBits = 12;
constexpr int kHllRegs = 1 << kHllBits;
// Longest probe sequence of the counting table. At load factor <= 0.5 linear
// probing stays far below it; reaching it counts as a full table.
constexpr uint64_t kMaxProbes = 4096;
// bin_kernel's shared memory: the chunk's records in bin order (keys), hot
// cache (key, count, first), bin counters, warp sums, record offsets, sketch
constexpr size_t kBinSmem = (size_t)kChunk * 8 + (size_t)kHotSlots * 16 + kBins * 4 +
                            kBinThreads / 32 * 4 + (size_t)kChunk * 2 + kHllRegs * 4;
constexpr int kWarpSpan = 1024;           // positions (or list entries) per warp chunk
static_assert(kChunk == kUnsortThreads / 32 * kWarpSpan, "a chunk is one unsort block's span");
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

// The table hash of a key. Its high bits pick the home slot (fastrange,
// Lemire 2019) and the bin, its low bits the shared-memory cache slots.
__device__ __forceinline__ uint64_t disc_hash(uint64_t key) { return fmix64(key ^ kDiscoverSeed); }

__device__ __forceinline__ uint64_t home_of(uint64_t h, uint64_t cap) { return __umul64hi(h, cap); }

__device__ __forceinline__ uint64_t slot_home(uint64_t key, uint64_t cap) {
  return home_of(disc_hash(key), cap);
}

// The table region a key's probe starts in: the top bits of the same hash, so
// that bin b holds the keys whose home slot lies in [b cap / kBins, (b + 1)
// cap / kBins].
__device__ __forceinline__ int bin_of(uint64_t h) { return (int)(h >> (64 - kBinBits)); }

// Sequence length L with its fastmod multiplier M = floor((2^64 - 1) / L) + 1:
// i mod L = high 64 bits of (M i mod 2^64) * L for every 32-bit i (Lemire,
// Kaser, Kurz 2019, "Faster remainder by direct computation").
struct SeqLen {
  uint32_t L;
  uint64_t M;
};

__device__ __forceinline__ uint32_t pos_in_seq(uint32_t i, SeqLen s) {
  return (uint32_t)__umul64hi(s.M * i, (uint64_t)s.L);
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
  const uint64_t limit = cap < kMaxProbes ? cap : kMaxProbes;
  for (uint64_t probe = 1; probe < limit; ++probe) {
    if (prev == 0 || prev == key) return (uint32_t)s;
    s = s + 1 == cap ? 0 : s + 1;
    prev = atomicCAS(&table[s].key, 0ull, (unsigned long long)key);
  }
  if (prev == 0 || prev == key) return (uint32_t)s;
  atomicExch(&err->table_full, 1);
  return kNone;
}

// Key of the window ending at position i for scan n, or 0 when the window is
// not counted: it crosses a sequence start, or a token is out of range (scan
// 2; err, when given, records it), or its prefix or suffix is not frequent
// (scan n >= 3: names[] holds the previous scan's names). names == nullptr for
// n = 2, where the prefix name is the previous token.
__device__ __forceinline__ uint64_t window_key(const int32_t* __restrict__ tok,
                                               const uint32_t* __restrict__ names, int64_t i,
                                               SeqLen L, int32_t n, int32_t vocab,
                                               DiscoverErr* err) {
  const int32_t t = tok[i];
  if (n == 2 && (t < 0 || t >= vocab)) {
    if (err) atomicExch(&err->token_range, 1);
    return 0;
  }
  if (pos_in_seq((uint32_t)i, L) < (uint32_t)(n - 1)) return 0;
  uint32_t pre;
  if (n == 2) {
    const int32_t tp = tok[i - 1];
    if (tp < 0 || tp >= vocab) return 0;
    pre = (uint32_t)tp;
  } else {
    pre = names[i - 1];
    if (pre == kNone || names[i] == kNone) return 0;
  }
  return ((uint64_t)(pre + 1u) << 32) | (uint32_t)t;
}

// (count, ~first) of key, or (0, 0) when the key is not in the table.
__device__ __forceinline__ uint2 lookup_slot(const CountSlot* __restrict__ table, uint64_t cap,
                                             uint64_t key) {
  uint64_t s = slot_home(key, cap);
  const uint64_t limit = cap < kMaxProbes ? cap : kMaxProbes;
  for (uint64_t probe = 0; probe < limit; ++probe) {
    const uint4 v = __ldg(reinterpret_cast<const uint4*>(table + s));
    const uint64_t k = (uint64_t)v.x | ((uint64_t)v.y << 32);
    if (k == key) return make_uint2(v.z, v.w);
    if (k == 0) break;
    s = s + 1 == cap ? 0 : s + 1;
  }
  return make_uint2(0u, 0u);
}

// Step 1a. Binning. Block b takes chunks of kChunk consecutive windows. A
// window whose key holds (or claims) its slot in the block's shared-memory
// cache of hot keys is counted there; the block keeps that cache for its
// whole run and adds it to the global table once at the end, so the hot keys
// of a Zipf corpus cost one global update per block. Every other window is a
// record {key, offset in chunk}, stored in the chunk's record area grouped by
// the key's bin (the top kBinBits bits of its table hash, i.e. the region of
// the table its probe starts in); off[chunk][bin] gives each group's start.
// Phase 1 counts the bins, phase 2 recomputes each window's key (its inputs
// are still in L2) and places the record in bin order in shared memory, and
// phase 3 writes the chunk's records out with coalesced stores.
__global__ void __launch_bounds__(kBinThreads, 1)
bin_kernel(const int32_t* __restrict__ tok, const uint32_t* __restrict__ names, int64_t N,
           SeqLen L, int32_t n, int32_t vocab, unsigned long long* __restrict__ rkey,
           uint16_t* __restrict__ rloc, uint32_t* __restrict__ off,
           CountSlot* __restrict__ hot_out, uint32_t* __restrict__ hll_out,
           unsigned long long* __restrict__ n_cand, unsigned long long* __restrict__ n_flush,
           DiscoverErr* err) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  auto* sk = reinterpret_cast<unsigned long long*>(smem_raw);             // [kChunk] in bin order
  auto* hkey = sk + kChunk;                                                // [kHotSlots]
  auto* hcnt = reinterpret_cast<uint32_t*>(hkey + kHotSlots);              // [kHotSlots]
  auto* hfirst = hcnt + kHotSlots;                                         // [kHotSlots]
  auto* bcnt = hfirst + kHotSlots;                                         // [kBins]
  auto* wsum = bcnt + kBins;                                               // [kBinThreads / 32]
  auto* sl = reinterpret_cast<uint16_t*>(wsum + kBinThreads / 32);         // [kChunk] in bin order
  auto* hll = reinterpret_cast<uint32_t*>(sl + kChunk);                    // [kHllRegs]
  for (int j = threadIdx.x; j < kHllRegs; j += kBinThreads) hll[j] = 0;
  for (int h = threadIdx.x; h < kHotSlots; h += kBinThreads) {
    hkey[h] = 0;
    hcnt[h] = 0;
    hfirst[h] = kNone;
  }
  for (int b = threadIdx.x; b < kBins; b += kBinThreads) bcnt[b] = 0;
  __syncthreads();
  unsigned long long my_cand = 0, my_flush = 0;
  const int64_t n_chunks = (N + kChunk - 1) / kChunk;
  constexpr int kPer = kChunk / kBinThreads;
  static_assert(kPer % kWin == 0, "whole batches of windows per thread");
  for (int64_t c = blockIdx.x; c < n_chunks; c += gridDim.x) {
    // phase 1: keys, hot cache, bin sizes (kWin windows' loads in flight)
#pragma unroll 1
    for (int u0 = 0; u0 < kPer; u0 += kWin) {
      uint64_t key[kWin];
#pragma unroll
      for (int u = 0; u < kWin; ++u) {
        const int64_t i = c * kChunk + (u0 + u) * kBinThreads + threadIdx.x;
        key[u] = i < N ? window_key(tok, names, i, L, n, vocab, err) : 0;
      }
#pragma unroll
      for (int u = 0; u < kWin; ++u) {
        if (!key[u]) continue;
        ++my_cand;
        const int64_t i = c * kChunk + (u0 + u) * kBinThreads + threadIdx.x;
        const uint32_t start = (uint32_t)(i - n + 1);
        const uint64_t hh = disc_hash(key[u]);
        // sketch: register from hash bits 11..22, rank = position of the
        // leftmost 1 among bits 23..63 (Flajolet et al. 2007)
        const uint32_t j = (uint32_t)(hh >> 11) & (kHllRegs - 1);
        const uint64_t wbits = hh >> (11 + kHllBits);
        const uint32_t rank = wbits ? (uint32_t)__clzll((long long)wbits) - (10 + kHllBits) : 42u;
        if (rank > hll[j]) atomicMax(&hll[j], rank);
        const uint32_t h = (uint32_t)hh & (kHotSlots - 1);
        const unsigned long long hp = atomicCAS(&hkey[h], 0ull, (unsigned long long)key[u]);
        if (hp == 0 || hp == key[u]) {
          atomicAdd(&hcnt[h], 1u);
          atomicMin(&hfirst[h], start);
        } else {
          atomicAdd(&bcnt[bin_of(hh)], 1u);
        }
      }
    }
    __syncthreads();
    // bin starts: exclusive scan of bcnt (one bin per thread), written to off
    static_assert(kBins == kBinThreads, "one bin per thread");
    uint32_t total;
    {
      const int lane = threadIdx.x & 31, warp = threadIdx.x / 32;
      const uint32_t a = bcnt[threadIdx.x];
      uint32_t incl = a;
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += v;
      }
      if (lane == 31) wsum[warp] = incl;
      __syncthreads();
      if (warp == 0) {
        uint32_t w = wsum[lane];
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t v = __shfl_up_sync(0xFFFFFFFFu, w, o);
          if (lane >= o) w += v;
        }
        wsum[lane] = w;   // inclusive over warps
      }
      __syncthreads();
      const uint32_t base = incl - a + (warp > 0 ? wsum[warp - 1] : 0u);
      total = wsum[kBinThreads / 32 - 1];
      uint32_t* o = off + c * (kBins + 1);
      o[threadIdx.x] = base;
      if (threadIdx.x == 0) o[kBins] = total;
      bcnt[threadIdx.x] = base;         // becomes the bin's write cursor
    }
    __syncthreads();
    // phase 2: every cold window's record to its place in bin order (a window
    // is cold exactly when its cache slot holds another key: claims made in
    // phase 1 are never undone)
#pragma unroll 1
    for (int u0 = 0; u0 < kPer; u0 += kWin) {
      uint64_t key[kWin];
#pragma unroll
      for (int u = 0; u < kWin; ++u) {
        const int64_t i = c * kChunk + (u0 + u) * kBinThreads + threadIdx.x;
        key[u] = i < N ? window_key(tok, names, i, L, n, vocab, nullptr) : 0;
      }
#pragma unroll
      for (int u = 0; u < kWin; ++u) {
        if (!key[u]) continue;
        const uint64_t hh = disc_hash(key[u]);
        if (hkey[(uint32_t)hh & (kHotSlots - 1)] == key[u]) continue;
        const uint32_t dst = atomicAdd(&bcnt[bin_of(hh)], 1u);
        sk[dst] = key[u];
        sl[dst] = (uint16_t)((u0 + u) * kBinThreads + threadIdx.x);
      }
    }
    __syncthreads();
    // phase 3: the chunk's records, coalesced
    my_flush += threadIdx.x == 0 ? total : 0u;
    for (uint32_t r = threadIdx.x; r < total; r += kBinThreads) {
      rkey[c * kChunk + r] = sk[r];
      rloc[c * kChunk + r] = sl[r];
    }
    bcnt[threadIdx.x] = 0;
    __syncthreads();
  }
  __syncthreads();
  for (int j = threadIdx.x; j < kHllRegs; j += kBinThreads)
    if (hll[j]) atomicMax(&hll_out[j], hll[j]);
  // the hot cache goes to this block's part of the hot list; hotflush_kernel
  // adds it to the table once the table is sized and zeroed
  for (int h = threadIdx.x; h < kHotSlots; h += kBinThreads) {
    CountSlot e;
    e.key = hkey[h];
    e.count = hcnt[h];
    e.first_inv = ~hfirst[h];
    hot_out[(int64_t)blockIdx.x * kHotSlots + h] = e;
  }
  for (int o = 16; o > 0; o >>= 1) {
    my_cand += __shfl_down_sync(0xFFFFFFFFu, my_cand, o);
    my_flush += __shfl_down_sync(0xFFFFFFFFu, my_flush, o);
  }
  if ((threadIdx.x & 31) == 0 && my_cand) atomicAdd(n_cand, my_cand);
  if ((threadIdx.x & 31) == 0 && my_flush) atomicAdd(n_flush, my_flush);
}

// Adds (cnt, first) of key to the global table, given the result prev of the
// CAS at its home slot; a full table is recorded in err.
__device__ __forceinline__ void table_add(CountSlot* __restrict__ table, uint64_t cap,
                                          uint64_t key, uint64_t home,
                                          unsigned long long prev, uint32_t cnt,
                                          uint32_t first, DiscoverErr* err) {
  const uint32_t g = probe_rest(table, cap, key, home, prev, err);
  if (g == kNone) return;
  atomicAdd(&table[g].count, cnt);
  atomicMax(&table[g].first_inv, ~first);
}

// Step 1a'. The binning blocks' hot-key caches added to the zeroed table:
// one thread per cache entry (key 0 = unused).
__global__ void __launch_bounds__(256)
hotflush_kernel(const CountSlot* __restrict__ hot, int64_t n_entries,
                CountSlot* __restrict__ table, uint64_t cap,
                unsigned long long* __restrict__ n_flush, DiscoverErr* err) {
  unsigned long long my_flush = 0;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n_entries;
       e += (int64_t)gridDim.x * blockDim.x) {
    const CountSlot v = hot[e];
    if (!v.key) continue;
    ++my_flush;
    const uint64_t home = slot_home(v.key, cap);
    const unsigned long long prev = atomicCAS(&table[home].key, 0ull, v.key);
    table_add(table, cap, v.key, home, prev, v.count, ~v.first_inv, err);
  }
  for (int o = 16; o > 0; o >>= 1) my_flush += __shfl_down_sync(0xFFFFFFFFu, my_flush, o);
  if ((threadIdx.x & 31) == 0 && my_flush) atomicAdd(n_flush, my_flush);
}

// Step 1b. Counting in table-region order. A work item is (bin, kItemChunks
// consecutive chunks); blocks take items in bin-major order from one ticket,
// so at any time all blocks update the same one or two regions of the table
// (cap / kBins slots each), which stay resident in L2. Warp w of the block
// reads the bin's groups of 32 of the item's chunks, one chunk per lane,
// flattened by a warp prefix sum so that every lane takes one record per
// step. A record is first counted in the block's shared-memory cache
// (direct-mapped, first key to claim a slot keeps it for the item); a record
// whose slot holds another key goes to the table at once. The cache is added
// to the table at the end of the item. A key that is frequent within its
// region thus costs one global update per item, not one per record: without
// the cache, its updates would all fall into the short time its region is
// being counted and serialize on one L2 slice.
__global__ void __launch_bounds__(kCntThreads)
bincount_kernel(const unsigned long long* __restrict__ rkey, const uint16_t* __restrict__ rloc,
                const uint32_t* __restrict__ off, int64_t n_chunks, int32_t n,
                CountSlot* __restrict__ table, uint64_t cap,
                unsigned long long* __restrict__ ticket, DiscoverErr* err) {
  extern __shared__ __align__(16) unsigned char cnt_smem[];
  auto* ckey = reinterpret_cast<unsigned long long*>(cnt_smem);           // [kCntSlots]
  auto* ccnt = reinterpret_cast<uint32_t*>(ckey + kCntSlots);              // [kCntSlots]
  auto* cfirst = ccnt + kCntSlots;                                          // [kCntSlots]
  __shared__ unsigned long long item_s[2];
  for (int h = threadIdx.x; h < kCntSlots; h += kCntThreads) {
    ckey[h] = 0;
    ccnt[h] = 0;
    cfirst[h] = kNone;
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x / 32;
  const int64_t n_groups = (n_chunks + kItemChunks - 1) / kItemChunks;
  const unsigned long long n_items = (unsigned long long)n_groups * kBins;
  if (threadIdx.x == 0) item_s[0] = atomicAdd(ticket, 1ull);
  __syncthreads();
  // Two barriers per item: after the records (the cache is complete) and
  // after the flush (the cache is empty, and the next ticket is in). Thread 0
  // takes the next ticket as the flush starts, so its round trip overlaps the
  // flush. It is not taken earlier: a block holding the next item while it
  // counts the current one widens the span of table regions being updated at
  // once, and the updates then miss L2 more often. item_s alternates between
  // two slots so that the next ticket never overwrites one still being read.
  for (int it = 0;; it ^= 1) {
    const unsigned long long item = item_s[it];
    if (item >= n_items) break;
    const int bin = (int)(item / n_groups);
    const int64_t c0 = (int64_t)(item % n_groups) * kItemChunks + warp * 32;
    uint32_t beg = 0, len = 0;
    if (c0 + lane < n_chunks) {
      const uint32_t* o = off + (c0 + lane) * (kBins + 1) + bin;
      beg = o[0];
      len = o[1] - beg;
    }
    uint32_t incl = len;
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += v;
    }
    const uint32_t excl = incl - len;
    const uint32_t total = __shfl_sync(0xFFFFFFFFu, incl, 31);
    for (uint32_t k0 = 0; k0 < total; k0 += 32 * kWin) {
      uint64_t key[kWin], home[kWin];
      unsigned long long prev[kWin];
      uint32_t start[kWin];
      bool cold[kWin];
#pragma unroll
      for (int u = 0; u < kWin; ++u) {
        const uint32_t k = k0 + u * 32 + lane;
        // j = the lane (chunk) whose group holds flattened record k
        int j = 0;
#pragma unroll
        for (int st = 16; st > 0; st >>= 1) {
          const uint32_t v = __shfl_sync(0xFFFFFFFFu, incl, j + st - 1);
          if (v <= k) j += st;
        }
        const uint32_t bj = __shfl_sync(0xFFFFFFFFu, beg, j);
        const uint32_t ej = __shfl_sync(0xFFFFFFFFu, excl, j);
        key[u] = 0;
        start[u] = 0;
        if (k < total) {
          const int64_t rec = (c0 + j) * kChunk + bj + (k - ej);
          key[u] = rkey[rec];
          start[u] = (uint32_t)((c0 + j) * kChunk + rloc[rec] - (n - 1));
        }
      }
#pragma unroll
      for (int u = 0; u < kWin; ++u) {
        cold[u] = false;
        if (!key[u]) continue;
        const uint64_t hh = disc_hash(key[u]);
        const uint32_t h = (uint32_t)hh & (kCntSlots - 1);
        const unsigned long long hp = atomicCAS(&ckey[h], 0ull, (unsigned long long)key[u]);
        if (hp == 0 || hp == key[u]) {
          atomicAdd(&ccnt[h], 1u);
          atomicMin(&cfirst[h], start[u]);
        } else {
          cold[u] = true;
          home[u] = home_of(hh, cap);
          prev[u] = atomicCAS(&table[home[u]].key, 0ull, (unsigned long long)key[u]);
        }
      }
#pragma unroll
      for (int u = 0; u < kWin; ++u)
        if (cold[u]) table_add(table, cap, key[u], home[u], prev[u], 1u, start[u], err);
    }
    __syncthreads();
    if (threadIdx.x == 0) item_s[it ^ 1] = atomicAdd(ticket, 1ull);
    // add the cache to the table and empty it; every probe of a batch is
    // issued before any result is used
    constexpr int kOwn = kCntSlots / kCntThreads;
    static_assert(kCntSlots % kCntThreads == 0 && kOwn % 4 == 0, "cache slots per thread");
#pragma unroll
    for (int h0 = 0; h0 < kOwn; h0 += 4) {
      unsigned long long key[4], prev[4];
      uint64_t home[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        key[k] = ckey[threadIdx.x + (h0 + k) * kCntThreads];
        home[k] = key[k] ? slot_home(key[k], cap) : 0;
        prev[k] = key[k] ? atomicCAS(&table[home[k]].key, 0ull, key[k]) : 0ull;
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int h = threadIdx.x + (h0 + k) * kCntThreads;
        if (!key[k]) continue;
        table_add(table, cap, key[k], home[k], prev[k], ccnt[h], cfirst[h], err);
        ckey[h] = 0;
        ccnt[h] = 0;
        cfirst[h] = kNone;
      }
    }
    __syncthreads();
  }
}

// A window's flag-pass result in 32 bits: the name its n-gram gets for the
// next scan (its first occurrence, < 2^30) or kNoName when the n-gram is not
// frequent; bit 30 = the window is its n-gram's first occurrence; bit 31 = it
// is also frequent (the n-gram enters the list of length n).
constexpr uint32_t kNoName = 0x3FFFFFFFu;

__device__ __forceinline__ uint32_t window_result(uint2 cf, uint32_t start, uint32_t min_count) {
  const bool first = ~cf.y == start;
  const bool eligible = cf.x >= min_count;
  return (eligible ? ~cf.y : kNoName) | (first ? 1u << 30 : 0u) |
         (first && eligible ? 1u << 31 : 0u);
}

// Step 2a. The records looked up in the finished table, in the same
// bin-major order as the counting (one region of the table in L2 at a time).
// A work item is (bin, 32 chunks) for one warp; each record's result goes to
// res[] at the record's index.
__global__ void __launch_bounds__(256)
flagbin_kernel(const unsigned long long* __restrict__ rkey, const uint16_t* __restrict__ rloc,
               const uint32_t* __restrict__ off, int64_t n_chunks, int32_t n,
               const CountSlot* __restrict__ table, uint64_t cap, uint32_t min_count,
               uint32_t* __restrict__ res, unsigned long long* __restrict__ ticket) {
  const int lane = threadIdx.x & 31;
  const int64_t n_groups = (n_chunks + 31) / 32;
  const unsigned long long n_items = (unsigned long long)n_groups * kBins;
  for (;;) {
    unsigned long long item = 0;
    if (lane == 0) item = atomicAdd(ticket, 1ull);
    item = __shfl_sync(0xFFFFFFFFu, item, 0);
    if (item >= n_items) break;
    const int bin = (int)(item / n_groups);
    const int64_t c0 = (int64_t)(item % n_groups) * 32;
    uint32_t beg = 0, len = 0;
    if (c0 + lane < n_chunks) {
      const uint32_t* o = off + (c0 + lane) * (kBins + 1) + bin;
      beg = o[0];
      len = o[1] - beg;
    }
    uint32_t incl = len;
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t v = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane >= o) incl += v;
    }
    const uint32_t excl = incl - len;
    const uint32_t total = __shfl_sync(0xFFFFFFFFu, incl, 31);
    for (uint32_t k0 = 0; k0 < total; k0 += 32 * kWin) {
      uint64_t key[kWin];
      int64_t rec[kWin];
      uint32_t start[kWin];
      uint4 v[kWin];
#pragma unroll
      for (int u = 0; u < kWin; ++u) {
        const uint32_t k = k0 + u * 32 + lane;
        int j = 0;
#pragma unroll
        for (int st = 16; st > 0; st >>= 1) {
          const uint32_t w = __shfl_sync(0xFFFFFFFFu, incl, j + st - 1);
          if (w <= k) j += st;
        }
        const uint32_t bj = __shfl_sync(0xFFFFFFFFu, beg, j);
        const uint32_t ej = __shfl_sync(0xFFFFFFFFu, excl, j);
        key[u] = 0;
        rec[u] = -1;
        start[u] = 0;
        if (k < total) {
          rec[u] = (c0 + j) * kChunk + bj + (k - ej);
          key[u] = rkey[rec[u]];
          start[u] = (uint32_t)((c0 + j) * kChunk + rloc[rec[u]] - (n - 1));
        }
      }
#pragma unroll
      for (int u = 0; u < kWin; ++u)
        v[u] = key[u] ? __ldg(reinterpret_cast<const uint4*>(table + slot_home(key[u], cap)))
                      : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
      for (int u = 0; u < kWin; ++u) {
        if (!key[u]) continue;
        const uint64_t k = (uint64_t)v[u].x | ((uint64_t)v[u].y << 32);
        const uint2 cf = k == key[u] ? make_uint2(v[u].z, v[u].w) : lookup_slot(table, cap, key[u]);
        res[rec[u]] = window_result(cf, start[u], min_count);
      }
    }
  }
}

// Step 2b. Back to position order, one chunk per block (8 warps of 1024
// positions): the chunk's record results are scattered into shared memory by
// window; a window without a record is either not counted (key 0) or was
// counted in a hot-key cache, and then looks its key up in the table (the hot
// keys' slots are few and stay in L2). One bit per position marks the first
// occurrences of frequent n-grams, counted per 1024 positions; each position
// also takes its n-gram's name for the next scan.
__global__ void __launch_bounds__(kUnsortThreads)
unsort_kernel(const uint32_t* __restrict__ res, const uint16_t* __restrict__ rloc,
              const uint32_t* __restrict__ off, const int32_t* __restrict__ tok,
              const uint32_t* __restrict__ names_in, int64_t N, SeqLen L, int32_t n,
              int32_t vocab, const CountSlot* __restrict__ table, uint64_t cap,
              uint32_t min_count, uint32_t* __restrict__ flags, uint32_t* __restrict__ chunk_cnt,
              uint32_t* __restrict__ name_out, unsigned long long* __restrict__ n_distinct,
              unsigned long long* __restrict__ n_named) {
  extern __shared__ uint32_t resw[];      // [kChunk]
  const int lane = threadIdx.x & 31, warp = threadIdx.x / 32;
  const int64_t n_chunks = (N + kChunk - 1) / kChunk;
  unsigned long long distinct = 0, named = 0;
  for (int64_t c = blockIdx.x; c < n_chunks; c += gridDim.x) {
    for (int w = threadIdx.x; w < kChunk; w += kUnsortThreads) resw[w] = kNone;
    __syncthreads();
    const uint32_t total = off[c * (kBins + 1) + kBins];
    for (uint32_t r = threadIdx.x; r < total; r += kUnsortThreads)
      resw[rloc[c * kChunk + r]] = res[c * kChunk + r];
    __syncthreads();
    const int64_t wc = c * (kChunk / kWarpSpan) + warp;     // this warp's 1024 positions
    uint32_t cnt = 0;
    constexpr int kBatch = 4;
    for (int it0 = 0; it0 < kWarpSpan / 32; it0 += kBatch) {
      uint32_t r[kBatch];
      uint64_t key[kBatch];
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        const int64_t i = wc * kWarpSpan + (it0 + b) * 32 + lane;
        r[b] = resw[warp * kWarpSpan + (it0 + b) * 32 + lane];
        key[b] = (r[b] == kNone && i < N) ? window_key(tok, names_in, i, L, n, vocab, nullptr)
                                          : 0;
      }
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        const int64_t i = wc * kWarpSpan + (it0 + b) * 32 + lane;
        if (key[b])
          r[b] = window_result(lookup_slot(table, cap, key[b]), (uint32_t)(i - n + 1), min_count);
        const bool has = r[b] != kNone;
        const uint32_t nm = r[b] & kNoName;
        if (name_out && i < N) {
          const bool eligible = has && nm != kNoName;
          name_out[i] = eligible ? nm : kNone;
          named += eligible;
        }
        const uint32_t word = __ballot_sync(0xFFFFFFFFu, has && (r[b] >> 31));
        const uint32_t dword = __ballot_sync(0xFFFFFFFFu, has && ((r[b] >> 30) & 1u));
        if (lane == 0 && wc * kWarpSpan + (it0 + b) * 32 < N)
          flags[(wc * kWarpSpan) / 32 + it0 + b] = word;
        cnt += __popc(word);
        distinct += __popc(dword);
      }
    }
    if (lane == 0 && wc * kWarpSpan < N) chunk_cnt[wc] = cnt;
    __syncthreads();
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

// Step 4. One warp per 1024 positions, in position order; each flagged
// window looks its count up again by key.
__global__ void __launch_bounds__(256)
assign_kernel(const uint32_t* __restrict__ flags, const unsigned long long* __restrict__ chunk_off,
              const int32_t* __restrict__ tok, const uint32_t* __restrict__ names_in, int64_t N,
              SeqLen L, int32_t n, int32_t vocab, const CountSlot* __restrict__ table,
              uint64_t cap, int32_t* __restrict__ list_tok, uint32_t* __restrict__ list_cnt) {
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
        const uint64_t key = window_key(tok, names_in, i, L, n, vocab, nullptr);
        list_cnt[id] = lookup_slot(table, cap, key).x;
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

// Pinned host memory that the call's small device-to-host reads land in (a
// copy into pageable memory is staged and synchronous in the driver).
struct HostStage {
  uint32_t hll[kHllRegs];
  unsigned long long counters[16];
  DiscoverErr err;
  unsigned int hist[256];
};

// Named buffers of a workspace.
enum Buf {
  kBufNames, kBufNamesNext, kBufRecKey, kBufRecLoc, kBufRecOff, kBufRecRes, kBufHot, kBufFlags,
  kBufChunkCnt, kBufChunkOff, kBufCounters, kBufErr, kBufTable, kBufHll,
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
  scone::HostStage* stage = nullptr;   // pinned, allocated on first use
  // counting-table slots per estimated distinct key: load factor 0.25. On the
  // 1.07e9-token corpus 4 beat 2.5 (longer probe chains) and 8 to 16 (more
  // table to clear and to miss in L2) by 2 to 4 ms per call.
  double table_slack = 4.0;
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
  scone::HostStage* host_stage() {
    if (!stage) {
      void* p = nullptr;
      if (cudaHostAlloc(&p, sizeof(scone::HostStage), cudaHostAllocDefault) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
      }
      stage = static_cast<scone::HostStage*>(p);
    }
    return stage;
  }
  ~scone_discover() {
    for (void* p : ptr)
      if (p) cudaFree(p);
    if (stage) cudaFreeHost(stage);
  }
};

namespace scone {
namespace {

// HyperLogLog estimate of the number of distinct keys from the sketch
// registers (Flajolet, Fusy, Gandouet, Meunier 2007), with linear counting
// for small cardinalities; 64-bit hashes need no large-range correction.
double hll_estimate(const uint32_t* reg, int n_regs) {
  const double m = (double)n_regs;
  double sum = 0.0;
  int zeros = 0;
  for (int j = 0; j < n_regs; ++j) {
    sum += std::ldexp(1.0, -(int)reg[j]);
    zeros += reg[j] == 0;
  }
  double e = 0.7213 / (1.0 + 1.079 / m) * m * m / sum;
  if (e <= 2.5 * m && zeros > 0) e = m * std::log(m / zeros);
  return e;
}

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

extern "C" int scone_discover_set_table_slack(scone_discover* ws, double slots_per_key) {
  if (!ws || !(slots_per_key > 0.0) || slots_per_key > 1e6) return SCONE_ERR_INVALID_ARG;
  ws->table_slack = slots_per_key;
  return SCONE_OK;
}

extern "C" int scone_discover_destroy(scone_discover* ws) {
  if (!ws) return SCONE_OK;
  DeviceGuard dg(ws->device);
  delete ws;
  return SCONE_OK;
}

extern "C" int scone_fgram_discover(scone_discover* ws, const int32_t* tok, int32_t B, int32_t L,
                                    int32_t vocab, int32_t K, int64_t S, int32_t min_count,
                                    int32_t* fgram_tok,
                                    uint8_t* fgram_len, uint32_t* fgram_count, int64_t* n_out,
                                    scone_discover_stats* stats, void* stream) {
  if (B < 0 || L < 0 || vocab < 1 || K < 2 || K > 8 || S < 0 || min_count < 1 || !n_out)
    return SCONE_ERR_INVALID_ARG;
  const int64_t N = (int64_t)B * L;
  if (N > (1ll << 30)) return SCONE_ERR_UNSUPPORTED;   // names and starts stay 30-bit
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
  cudaEvent_t ev_c0[9], ev_b1[9], ev_k0[9], ev_c1[9], ev_f1[9], ev_s0[9], ev_s1[9];
  for (int n = 0; n <= 8; ++n) {
    ev_c0[n] = evs.make();
    ev_b1[n] = evs.make();
    ev_k0[n] = evs.make();
    ev_c1[n] = evs.make();
    ev_f1[n] = evs.make();
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
  const int64_t n_chunks = (N + kChunk - 1) / kChunk;
  // names ping-pong between scans: scan n reads the previous scan's names and
  // writes its own (scan 2 writes names[1], scan 3 names[0], ...)
  uint32_t* names[2] = {K > 3 ? static_cast<uint32_t*>(get(kBufNames, (size_t)N * 4)) : nullptr,
                        K > 2 ? static_cast<uint32_t*>(get(kBufNamesNext, (size_t)N * 4))
                              : nullptr};
  auto* rkey = static_cast<unsigned long long*>(get(kBufRecKey, (size_t)n_chunks * kChunk * 8));
  auto* rloc = static_cast<uint16_t*>(get(kBufRecLoc, (size_t)n_chunks * kChunk * 2));
  auto* roff = static_cast<uint32_t*>(get(kBufRecOff, (size_t)n_chunks * (kBins + 1) * 4));
  auto* rres = static_cast<uint32_t*>(get(kBufRecRes, (size_t)n_chunks * kChunk * 4));
  auto* flags = static_cast<uint32_t*>(get(kBufFlags, (size_t)n_words * 4));
  auto* chunk_cnt = static_cast<uint32_t*>(get(kBufChunkCnt, (size_t)n_wchunks * 4));
  auto* chunk_off = static_cast<unsigned long long*>(get(kBufChunkOff, (size_t)n_wchunks * 8));
  // counters: 0 candidates, 1 distinct, 2 frequent, 3 named, 4 and 5 selection
  // totals, 6 binned windows, 7 and 8 the tickets of the two bin-major passes,
  // 9 hot-cache entries added to the table
  constexpr int kCounters = 16;
  auto* counters = static_cast<unsigned long long*>(get(kBufCounters, kCounters * 8));
  auto* d_err = static_cast<DiscoverErr*>(get(kBufErr, sizeof(DiscoverErr)));
  auto* hll = static_cast<uint32_t*>(get(kBufHll, kHllRegs * sizeof(uint32_t)));
  HostStage* hs = ws->host_stage();
  if (nomem || !hs) return SCONE_ERR_NOMEM;
  if (cudaMemsetAsync(d_err, 0, sizeof(DiscoverErr), s) != cudaSuccess) return SCONE_ERR_CUDA;
  if (cudaFuncSetAttribute((const void*)bin_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)kBinSmem) != cudaSuccess)
    return SCONE_ERR_CUDA;
  if (cudaFuncSetAttribute((const void*)unsort_kernel,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, kChunk * 4) != cudaSuccess)
    return SCONE_ERR_CUDA;
  const int g_bin = grid_for((const void*)bin_kernel, kBinThreads, kBinSmem, n_chunks);
  auto* hot =
      static_cast<CountSlot*>(get(kBufHot, (size_t)g_bin * kHotSlots * sizeof(CountSlot)));
  if (nomem) return SCONE_ERR_NOMEM;
  const int g_hot = grid_for((const void*)hotflush_kernel, 256, 0,
                             ((int64_t)g_bin * kHotSlots + 255) / 256);
  if (cudaFuncSetAttribute((const void*)bincount_kernel,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kCntSmem) !=
      cudaSuccess)
    return SCONE_ERR_CUDA;
  const int g_cnt = grid_for((const void*)bincount_kernel, kCntThreads, kCntSmem,
                             (n_chunks + kItemChunks - 1) / kItemChunks * kBins);
  const int g_flag = grid_for((const void*)flagbin_kernel, 256, 0,
                              ((n_chunks + 31) / 32 * kBins + 7) / 8);
  const int g_uns = grid_for((const void*)unsort_kernel, kUnsortThreads, kChunk * 4, n_chunks);
  const int gw = grid_for((const void*)assign_kernel, 256, 0, (n_wchunks + 7) / 8);
  int cur = 0;                      // names[cur]: the names of the previous scan
  const SeqLen Ls{(uint32_t)L, ~0ull / (uint64_t)L + 1};

  std::vector<uint32_t*> list_cnt(K + 1, nullptr);
  std::vector<int32_t*> list_tok(K + 1, nullptr);
  std::vector<int64_t> list_size(K + 1, 0);

  int64_t cand_bound = (int64_t)B * (L > 0 ? L - 1 : 0);   // windows of length 2
  for (int n = 2; n <= K; ++n) {
    if (cand_bound == 0 && n > 2) break;   // scan 2 always runs: it checks every token
    if (ev_s0[n]) cudaEventRecord(ev_s0[n], s);
    if (cudaMemsetAsync(counters, 0, kCounters * sizeof(unsigned long long), s) != cudaSuccess ||
        cudaMemsetAsync(hll, 0, kHllRegs * sizeof(uint32_t), s) != cudaSuccess)
      return SCONE_ERR_CUDA;

    if (ev_c0[n]) cudaEventRecord(ev_c0[n], s);
    const uint32_t* names_in = n == 2 ? nullptr : names[cur];
    uint32_t* names_out = n < K ? names[cur ^ 1] : nullptr;
    bin_kernel<<<g_bin, kBinThreads, kBinSmem, s>>>(tok, names_in, N, Ls, n, vocab, rkey, rloc,
                                                    roff, hot, hll, counters + 0, counters + 6,
                                                    d_err);
    if (ev_b1[n]) cudaEventRecord(ev_b1[n], s);
    if (cudaGetLastError() != cudaSuccess) return SCONE_ERR_CUDA;
    // size the table from the sketch of the distinct keys
    if (cudaMemcpyAsync(hs->hll, hll, kHllRegs * sizeof(uint32_t), cudaMemcpyDeviceToHost, s) !=
            cudaSuccess ||
        cudaMemcpyAsync(hs->counters, counters, sizeof(unsigned long long),
                        cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
      return SCONE_ERR_CUDA;
    const unsigned long long n_cand = hs->counters[0];
    const double est = hll_estimate(hs->hll, kHllRegs);
    // at most one distinct n-gram per counted window: load factor <= 0.5
    const uint64_t worst = 2 * n_cand > 64 ? 2 * n_cand : 64;
    const double want = std::ceil(ws->table_slack * est);
    uint64_t cap = want < 64.0 ? 64 : (want >= (double)worst ? worst : (uint64_t)want);
    st.estimate[n] = (int64_t)std::llround(est);

    unsigned long long h[10];
    DiscoverErr herr;
    CountSlot* table = nullptr;
    for (int attempt = 0;; ++attempt) {
      table = static_cast<CountSlot*>(get(kBufTable, (size_t)cap * sizeof(CountSlot)));
      if (nomem) return SCONE_ERR_NOMEM;
      if (ev_k0[n]) cudaEventRecord(ev_k0[n], s);
      if (cudaMemsetAsync(table, 0, cap * sizeof(CountSlot), s) != cudaSuccess)
        return SCONE_ERR_CUDA;
      hotflush_kernel<<<g_hot, 256, 0, s>>>(hot, (int64_t)g_bin * kHotSlots, table, cap,
                                            counters + 9, d_err);
      bincount_kernel<<<g_cnt, kCntThreads, kCntSmem, s>>>(rkey, rloc, roff, n_chunks, n, table,
                                                           cap, counters + 7, d_err);
      if (ev_c1[n]) cudaEventRecord(ev_c1[n], s);
      flagbin_kernel<<<g_flag, 256, 0, s>>>(rkey, rloc, roff, n_chunks, n, table, cap,
                                            (uint32_t)min_count, rres, counters + 8);
      unsort_kernel<<<g_uns, kUnsortThreads, kChunk * 4, s>>>(
          rres, rloc, roff, tok, names_in, N, Ls, n, vocab, table, cap, (uint32_t)min_count,
          flags, chunk_cnt, names_out, counters + 1, counters + 3);
      if (ev_f1[n]) cudaEventRecord(ev_f1[n], s);
      scan_kernel<<<1, kScanThreads, 0, s>>>(chunk_cnt, chunk_off, n_wchunks, counters + 2);
      if (cudaGetLastError() != cudaSuccess) return SCONE_ERR_CUDA;
      if (cudaMemcpyAsync(hs->counters, counters, sizeof(h), cudaMemcpyDeviceToHost, s) !=
              cudaSuccess ||
          cudaMemcpyAsync(&hs->err, d_err, sizeof(herr), cudaMemcpyDeviceToHost, s) !=
              cudaSuccess ||
          cudaStreamSynchronize(s) != cudaSuccess)
        return SCONE_ERR_CUDA;
      std::memcpy(h, hs->counters, sizeof(h));
      herr = hs->err;
      if (herr.token_range) return SCONE_ERR_TOKEN_RANGE;
      if (!herr.table_full) break;
      if (cap >= worst) return SCONE_ERR_TABLE_FULL;
      // the sketch underestimated: count and flag again in a worst-case table
      // (the binned records stay valid)
      ++st.table_rebuilds;
      cap = worst;
      if (cudaMemsetAsync(d_err, 0, sizeof(DiscoverErr), s) != cudaSuccess ||
          cudaMemsetAsync(counters + 1, 0, 3 * sizeof(unsigned long long), s) != cudaSuccess ||
          cudaMemsetAsync(counters + 7, 0, 3 * sizeof(unsigned long long), s) != cudaSuccess)
        return SCONE_ERR_CUDA;
    }
    st.candidates[n] = (int64_t)h[0];
    st.distinct[n] = (int64_t)h[1];
    st.frequent[n] = (int64_t)h[2];
    st.flushes[n] = (int64_t)(h[6] + h[9]);
    st.ms_bin[n] = elapsed_ms(ev_c0[n], ev_b1[n]);
    st.ms_count[n] = elapsed_ms(ev_k0[n], ev_c1[n]);
    st.ms_flag[n] = elapsed_ms(ev_c1[n], ev_f1[n]);
    const int64_t M = (int64_t)h[2];
    list_size[n] = M;
    list_cnt[n] = static_cast<uint32_t*>(get(kBufListCnt + n, (size_t)M * 4));
    list_tok[n] = static_cast<int32_t*>(get(kBufListTok + n, (size_t)M * n * 4));
    if (nomem) return SCONE_ERR_NOMEM;
    if (M > 0)
      assign_kernel<<<gw, 256, 0, s>>>(flags, chunk_off, tok, names_in, N, Ls, n, vocab, table,
                                       cap, list_tok[n], list_cnt[n]);
    // windows of eligible n-grams bound the windows of the next scan
    cand_bound = n < K && M > 0 ? (int64_t)h[3] : 0;
    cur ^= 1;
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
      const unsigned int* hh = hs->hist;
      if (cudaMemsetAsync(hist, 0, 256 * sizeof(unsigned int), s) != cudaSuccess)
        return SCONE_ERR_CUDA;
      hist_kernel<<<hg, 256, 0, s>>>(ls, shift, mask, prefix, hist);
      if (cudaGetLastError() != cudaSuccess ||
          cudaMemcpyAsync(hs->hist, hist, 256 * sizeof(unsigned int), cudaMemcpyDeviceToHost,
                          s) != cudaSuccess ||
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
