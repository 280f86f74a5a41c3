// f-gram table build, lifetime and status (C ABI).
//
// Build (Sec. 2: "a hash dictionary that maps f-grams to matrix indices") of
// the bucketized cuckoo table described in scone_device.cuh:
//   1. the slot array is set to all ones (every row word = empty);
//   2. one thread per f-gram places its row: it tries to claim an empty slot
//      of either candidate bucket with a 32-bit atomicCAS on the row word;
//      if both buckets are full it swaps its row into one of them with
//      atomicExch and carries the evicted row to that row's other bucket
//      (parallel cuckoo insertion, Alcantara et al. 2009). Rows are compared
//      through the device copy of the input list, which is immutable during
//      the build, so no thread ever waits on another. An eviction chain
//      longer than kMaxKicks fails the attempt, which is retried from an
//      empty table with a new hash seed;
//   3. one thread per slot writes the packed key of the row it holds;
//   4. one thread per f-gram looks its key up in the finished table: it must
//      find its own row. Finding another row means the list holds the same
//      n-gram twice (also when two copies raced past the checks in step 2).
// With a suffix index (scone_device.cuh) the entries placed are the listed
// f-grams followed by the marker n-grams computed on the host
// (scone_suffix.cu); step 3 writes each slot's final row word (row and
// extension bit, or the marker word) and step 4 checks those words.

#include <sys/mman.h>
#include <unistd.h>

#include <cmath>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <new>
#include <thread>
#include <vector>

#include "scone_device.cuh"
#include "scone_host.h"

namespace scone {

namespace {

constexpr int kMaxKicks = 512;      // eviction steps before an attempt is abandoned
constexpr int kMaxAttempts = 8;     // hash seeds tried per build

struct BuildFlags {
  int duplicate;
  int full;        // an eviction chain exceeded kMaxKicks, or a row was lost
  int max_kicks;   // most evictions one insert needed
};

template <int FMT>
__device__ __forceinline__ KeyBits<Fmt<FMT>::kWords> key_of_listed(const int32_t* ftok,
                                                                    const uint8_t* flen,
                                                                    int64_t r, int K, int bits) {
  constexpr int NW = Fmt<FMT>::kWords;
  KeyBits<NW> k;
#pragma unroll
  for (int q = 0; q < NW; ++q) k.w[q] = 0;
  const int n = flen[r];
  const int32_t* g = ftok + r * K;
  k.w[0] = (uint32_t)g[n - 1];
  for (int j = 1; j < n; ++j) put_field<NW>(k, j * bits, (uint32_t)g[n - 1 - j], bits);
  put_len<FMT>(k, n);
  return k;
}

__device__ __forceinline__ bool same_fgram(const int32_t* ftok, const uint8_t* flen, int64_t a,
                                           int64_t b, int K) {
  if (flen[a] != flen[b]) return false;
  for (int j = 0; j < flen[a]; ++j)
    if (ftok[a * K + j] != ftok[b * K + j]) return false;
  return true;
}

// The row word of slot s of bucket q (the upper half of the slot's last 8 bytes).
template <int FMT>
__device__ __forceinline__ unsigned int* row_word(uint8_t* slots, uint64_t q, int s) {
  constexpr int SLOT = Fmt<FMT>::kSlotBytes;
  return reinterpret_cast<unsigned int*>(slots + q * bucket_bytes<FMT>() + s * SLOT + SLOT - 4);
}

template <int FMT>
__global__ void insert_kernel(uint8_t* slots, uint64_t n_buckets, uint64_t seed,
                              const int32_t* ftok, const uint8_t* flen, int64_t n, int K, int bits,
                              BuildFlags* flags) {
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n;
       r += (int64_t)gridDim.x * blockDim.x) {
    unsigned int cur = (unsigned int)r;   // the row this thread is placing
    uint64_t from = ~0ull;                // the bucket `cur` was just evicted from
    bool done = false;
    int kick = 0;
    for (; kick <= kMaxKicks && !done; ++kick) {
      const auto k = key_of_listed<FMT>(ftok, flen, (int64_t)cur, K, bits);
      uint64_t b[2];
      cuckoo_buckets(key_hash<FMT>(k, seed), n_buckets, &b[0], &b[1]);
#pragma unroll
      for (int i = 0; i < 2 && !done; ++i) {
#pragma unroll
        for (int s = 0; s < kSlotsPerBucket && !done; ++s) {
          const unsigned int old = atomicCAS(row_word<FMT>(slots, b[i], s), kEmptyRow, cur);
          if (old == kEmptyRow) {
            done = true;
          } else if (same_fgram(ftok, flen, (int64_t)old, (int64_t)cur, K)) {
            atomicExch(&flags->duplicate, 1);
            done = true;
          }
        }
      }
      if (done || kick == kMaxKicks) break;
      // both buckets full: take a slot of the bucket `cur` did not come from
      const uint64_t vb = b[0] == from ? b[1] : (b[1] == from ? b[0] : b[kick & 1]);
      const int vs = (int)((cur ^ (unsigned int)kick) & 1);
      const unsigned int old = atomicExch(row_word<FMT>(slots, vb, vs), cur);
      if (old == kEmptyRow) {
        done = true;
      } else if (same_fgram(ftok, flen, (int64_t)old, (int64_t)cur, K)) {
        atomicExch(&flags->duplicate, 1);
        done = true;
      } else {
        cur = old;
        from = vb;
      }
    }
    if (done) {
      atomicMax(&flags->max_kicks, kick);
    } else {
      atomicExch(&flags->full, 1);
    }
  }
}

// The final row word of entry e: a listed f-gram's row (with its extension
// bit when ext is given), or the marker word for the entries past n_real.
__device__ __forceinline__ uint32_t entry_word(uint32_t e, const uint8_t* ext, int64_t n_real) {
  if ((int64_t)e >= n_real) return kMarkerWord;
  return e | (ext && ext[e] ? kExtBit : 0u);
}

template <int FMT>
__global__ void fill_keys_kernel(uint8_t* slots, uint64_t n_slots, const int32_t* ftok,
                                 const uint8_t* flen, int K, int bits, const uint8_t* ext,
                                 int64_t n_real) {
  constexpr int SLOT = Fmt<FMT>::kSlotBytes;
  constexpr int NW = Fmt<FMT>::kWords;
  for (uint64_t s = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; s < n_slots;
       s += (uint64_t)gridDim.x * blockDim.x) {
    uint64_t* w = reinterpret_cast<uint64_t*>(slots + s * SLOT);
    const uint32_t row = (uint32_t)(w[NW - 1] >> 32);
    if (row == kEmptyRow) continue;
    const auto k = key_of_listed<FMT>(ftok, flen, (int64_t)row, K, bits);
#pragma unroll
    for (int q = 0; q < NW - 1; ++q) w[q] = k.w[q];
    w[NW - 1] = (uint64_t)(uint32_t)k.w[NW - 1] |
                ((uint64_t)entry_word(row, ext, n_real) << 32);
  }
}

// The row word stored with the key (first bucket, then the second if the
// first is full without it), or kEmptyRow.
template <int FMT>
__device__ __forceinline__ uint32_t lookup_word(const TableView& t,
                                                const KeyBits<Fmt<FMT>::kWords>& k) {
  uint64_t b1, b2;
  cuckoo_buckets(key_hash<FMT>(k, t.hash_seed), t.n_buckets, &b1, &b2);
  const BucketData<FMT> v1 = ld_bucket_data<FMT>(t, b1);
  const uint32_t w = find_word_in_bucket<FMT>(v1, k);
  if (w != kEmptyRow || !bucket_full<FMT>(v1)) return w;
  return find_word_in_bucket<FMT>(ld_bucket_data<FMT>(t, b2), k);
}

template <int FMT>
__global__ void verify_kernel(TableView t, const int32_t* ftok, const uint8_t* flen, int64_t n,
                              int K, const uint8_t* ext, int64_t n_real, BuildFlags* flags) {
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < n;
       r += (int64_t)gridDim.x * blockDim.x) {
    const auto k = key_of_listed<FMT>(ftok, flen, r, K, t.bits);
    const uint32_t found = lookup_word<FMT>(t, k);
    if (found == kEmptyRow) atomicExch(&flags->full, 1);     // lost in a failed chain
    else if (found != entry_word((uint32_t)r, ext, n_real)) atomicExch(&flags->duplicate, 1);
  }
}

int grid_for(int64_t n, int threads) {
  int dev = 0, sms = 1;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t g = (n + threads - 1) / threads;
  const int64_t cap = (int64_t)sms * 32;
  if (g > cap) g = cap;
  return g < 1 ? 1 : (int)g;
}

int bits_for_vocab(int32_t vocab) {
  int b = 0;
  while (b < 31 && ((int64_t)1 << b) < (int64_t)vocab) ++b;
  return b < 1 ? 1 : b;
}

bool is_device_accessible(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}


// Steps 1-4 of the build into t->slots for n entries already on the device:
// the listed f-grams (the first n_real) and then the markers; d_ext (or
// NULL) holds the f-grams' extension bits. Tries kMaxAttempts hash seeds;
// sets t->view.hash_seed and *out_flags. Synchronizes the stream. Returns
// SCONE_OK, DUPLICATE_FGRAM, TABLE_FULL or CUDA.
int build_slots(scone_table* t, const int32_t* d_tok, const uint8_t* d_len, const uint8_t* d_ext,
                int64_t n_real, BuildFlags* d_flags, int64_t n, cudaStream_t s,
                BuildFlags* out_flags) {
  const uint64_t nb = (uint64_t)t->info.n_buckets;
  const uint64_t n_slots = (uint64_t)t->info.n_slots;
  const int K = t->view.K, bits = t->view.bits;
  const size_t bytes = (size_t)t->info.table_bytes;
  const int th = 256;
  BuildFlags flags = {0, 0, 0};
  for (int attempt = 0; attempt < kMaxAttempts; ++attempt) {
    const uint64_t seed = kHashSeed + (uint64_t)attempt * 0x9E3779B97F4A7C15ull;
    flags = {0, 0, 0};
    if (cudaMemsetAsync(t->slots, 0xFF, bytes, s) != cudaSuccess) return SCONE_ERR_CUDA;
    if (n > 0) {
      if (cudaMemsetAsync(d_flags, 0, sizeof(BuildFlags), s) != cudaSuccess)
        return SCONE_ERR_CUDA;
      TableView v = t->view;
      v.hash_seed = seed;
      v.probe_limit = 2;
      if (t->fmt == FMT16) {
        insert_kernel<FMT16><<<grid_for(n, th), th, 0, s>>>(t->slots, nb, seed, d_tok, d_len, n,
                                                            K, bits, d_flags);
        fill_keys_kernel<FMT16><<<grid_for((int64_t)n_slots, th), th, 0, s>>>(
            t->slots, n_slots, d_tok, d_len, K, bits, d_ext, n_real);
        verify_kernel<FMT16><<<grid_for(n, th), th, 0, s>>>(v, d_tok, d_len, n, K, d_ext, n_real,
                                                          d_flags);
      } else {
        insert_kernel<FMT32><<<grid_for(n, th), th, 0, s>>>(t->slots, nb, seed, d_tok, d_len, n,
                                                            K, bits, d_flags);
        fill_keys_kernel<FMT32><<<grid_for((int64_t)n_slots, th), th, 0, s>>>(
            t->slots, n_slots, d_tok, d_len, K, bits, d_ext, n_real);
        verify_kernel<FMT32><<<grid_for(n, th), th, 0, s>>>(v, d_tok, d_len, n, K, d_ext, n_real,
                                                          d_flags);
      }
      if (cudaGetLastError() != cudaSuccess ||
          cudaMemcpyAsync(&flags, d_flags, sizeof(BuildFlags), cudaMemcpyDeviceToHost, s) !=
              cudaSuccess)
        return SCONE_ERR_CUDA;
    }
    if (cudaStreamSynchronize(s) != cudaSuccess) return SCONE_ERR_CUDA;
    *out_flags = flags;
    if (flags.duplicate) return SCONE_ERR_DUPLICATE_FGRAM;
    if (!flags.full) {
      t->view.hash_seed = seed;
      return SCONE_OK;
    }
  }
  return SCONE_ERR_TABLE_FULL;
}
}  // namespace

}  // namespace scone

using namespace scone;

extern "C" int scone_table_build(const int32_t* fgram_tok, const uint8_t* fgram_len,
                                 int64_t n_fgrams, int32_t K, int32_t vocab, int32_t d,
                                 const scone_bf16* F, int32_t F_location, const scone_bf16* T,
                                 float load_factor, void* stream, scone_table** out) {
  if (!out) return SCONE_ERR_INVALID_ARG;
  *out = nullptr;
  if (n_fgrams < 0 || n_fgrams > 0x7FFFFFFELL || K < 2 || K > 8 || vocab < 1 || d < 1 || !T)
    return SCONE_ERR_INVALID_ARG;
  if (n_fgrams > 0 && (!fgram_tok || !fgram_len || !F)) return SCONE_ERR_INVALID_ARG;
  if (F_location != SCONE_ROWS_DEVICE && F_location != SCONE_ROWS_HOST_MAPPED)
    return SCONE_ERR_INVALID_ARG;
  if (load_factor == 0.0f) load_factor = 0.5f;
  if (!(load_factor > 0.0f && load_factor <= 0.85f)) return SCONE_ERR_INVALID_ARG;
  const int bits = bits_for_vocab(vocab);
  const int key_bits = K * bits + 4;
  int fmt;
  if (K * bits <= 92) {
    fmt = FMT16;
  } else if (K * bits <= 220) {
    fmt = FMT32;
  } else {
    return SCONE_ERR_UNSUPPORTED;
  }
  // host validation of the list: lengths in [2, K], tokens in [0, vocab)
  for (int64_t r = 0; r < n_fgrams; ++r) {
    const int n = fgram_len[r];
    if (n < 2 || n > K) return SCONE_ERR_INVALID_ARG;
    for (int j = 0; j < n; ++j)
      if (fgram_tok[r * K + j] < 0 || fgram_tok[r * K + j] >= vocab) return SCONE_ERR_INVALID_ARG;
  }
  // the suffix index: extension bits of the listed f-grams and the markers
  SuffixIndex si;
  const bool indexed = wants_suffix_index(fmt, K);
  if (indexed && n_fgrams > 0) {
    const int rc = suffix_index(fgram_tok, fgram_len, n_fgrams, K, &si);
    if (rc != SCONE_OK) return rc;
  }
  const int64_t n_entries = n_fgrams + si.n_markers;
  if (!is_device_accessible(T)) return SCONE_ERR_INVALID_ARG;
  const uint16_t* F_dev = reinterpret_cast<const uint16_t*>(F);
  if (n_fgrams > 0) {
    if (F_location == SCONE_ROWS_DEVICE) {
      if (!is_device_accessible(F)) return SCONE_ERR_INVALID_ARG;
    } else {
      void* dp = nullptr;
      if (cudaHostGetDevicePointer(&dp, const_cast<scone_bf16*>(F), 0) != cudaSuccess || !dp) {
        cudaGetLastError();
        return SCONE_ERR_INVALID_ARG;
      }
      F_dev = reinterpret_cast<const uint16_t*>(dp);
    }
  }

  int64_t n_slots = (int64_t)std::ceil((double)n_entries / (double)load_factor);
  if (n_slots < n_entries + 1) n_slots = n_entries + 1;
  int64_t n_buckets = (n_slots + kSlotsPerBucket - 1) / kSlotsPerBucket;
  if (n_buckets < 2) n_buckets = 2;   // two distinct candidate buckets
  n_slots = n_buckets * kSlotsPerBucket;
  const int64_t bucket = fmt == FMT16 ? bucket_bytes<FMT16>() : bucket_bytes<FMT32>();

  scone_table* t = new (std::nothrow) scone_table();
  if (!t) return SCONE_ERR_NOMEM;
  cudaGetDevice(&t->device);
  cudaStream_t s = (cudaStream_t)stream;
  if (cudaMalloc(&t->slots, (size_t)(n_buckets * bucket)) != cudaSuccess ||
      cudaMalloc(&t->status, sizeof(int)) != cudaSuccess ||
      cudaMalloc(&t->zero_row, (size_t)d * 2) != cudaSuccess) {
    cudaGetLastError();
    scone_table_destroy(t);
    return SCONE_ERR_NOMEM;
  }
  // the status mirror is an optimisation: without it scone_status copies the
  // word. Word 0 is the copy the recording kernel writes, word 1 receives the
  // status word when scone_status fetches it.
  void* mirror = nullptr;
  if (cudaHostAlloc(&mirror, 2 * sizeof(int), cudaHostAllocMapped) == cudaSuccess) {
    t->status_host = static_cast<int*>(mirror);
    t->status_host[0] = 0;
    t->status_host[1] = 0;
    void* dp = nullptr;
    if (cudaHostGetDevicePointer(&dp, mirror, 0) == cudaSuccess) {
      t->status_host_dev = static_cast<int*>(dp);
    } else {
      cudaFreeHost(mirror);
      t->status_host = nullptr;
    }
  }
  cudaGetLastError();
  t->fmt = fmt;
  TableView& v = t->view;
  v.slots = t->slots;
  v.n_buckets = (uint64_t)n_buckets;
  v.hash_seed = kHashSeed;
  v.probe_limit = 2;
  v.n_fgrams = n_fgrams;
  v.F = F_dev;
  v.T = reinterpret_cast<const uint16_t*>(T);
  v.status = t->status;
  v.status_mirror = t->status_host_dev;   // NULL without a mapped mirror
  v.K = K;
  v.bits = bits;
  v.vocab = vocab;
  v.d = d;
  v.suffix_index = indexed ? 1 : 0;
  scone_table_info& in = t->info;
  in.n_fgrams = n_fgrams;
  in.n_slots = n_slots;
  in.n_buckets = n_buckets;
  in.slot_bytes = fmt == FMT16 ? Fmt<FMT16>::kSlotBytes : Fmt<FMT32>::kSlotBytes;
  in.key_bits = key_bits;
  in.bits_per_token = bits;
  in.K = K;
  in.vocab = vocab;
  in.d = d;
  in.F_location = F_location;
  in.table_bytes = n_buckets * bucket;
  in.F_bytes = n_fgrams * (int64_t)d * 2;
  in.T_bytes = (int64_t)vocab * d * 2;
  in.n_markers = si.n_markers;
  in.suffix_index = v.suffix_index;

  int rc = SCONE_OK;
  int32_t* d_tok = nullptr;
  uint8_t* d_len = nullptr;
  uint8_t* d_ext = nullptr;
  BuildFlags* d_flags = nullptr;
  BuildFlags flags = {0, 0, 0};
  do {
    if (cudaMemsetAsync(t->status, 0, sizeof(int), s) != cudaSuccess ||
        cudaMemsetAsync(t->zero_row, 0, (size_t)d * 2, s) != cudaSuccess) {
      rc = SCONE_ERR_CUDA;
      break;
    }
    if (n_entries > 0) {
      // entries: the listed f-grams, then the markers
      const int64_t nm = si.n_markers;
      if (cudaMalloc(&d_tok, (size_t)n_entries * K * sizeof(int32_t)) != cudaSuccess ||
          cudaMalloc(&d_len, (size_t)n_entries) != cudaSuccess ||
          (indexed && cudaMalloc(&d_ext, (size_t)n_fgrams) != cudaSuccess) ||
          cudaMalloc(&d_flags, sizeof(BuildFlags)) != cudaSuccess) {
        rc = SCONE_ERR_NOMEM;
        break;
      }
      if (cudaMemcpyAsync(d_tok, fgram_tok, (size_t)n_fgrams * K * sizeof(int32_t),
                          cudaMemcpyHostToDevice, s) != cudaSuccess ||
          cudaMemcpyAsync(d_len, fgram_len, (size_t)n_fgrams, cudaMemcpyHostToDevice, s) !=
              cudaSuccess ||
          (nm > 0 && cudaMemcpyAsync(d_tok + n_fgrams * K, si.marker_tok.data(),
                                     (size_t)nm * K * sizeof(int32_t), cudaMemcpyHostToDevice,
                                     s) != cudaSuccess) ||
          (nm > 0 && cudaMemcpyAsync(d_len + n_fgrams, si.marker_len.data(), (size_t)nm,
                                     cudaMemcpyHostToDevice, s) != cudaSuccess) ||
          (d_ext && cudaMemcpyAsync(d_ext, si.ext.data(), (size_t)n_fgrams,
                                    cudaMemcpyHostToDevice, s) != cudaSuccess)) {
        rc = SCONE_ERR_CUDA;
        break;
      }
    }
    // (build_slots synchronizes the stream, so the host vectors outlive the copies)
    rc = build_slots(t, d_tok, d_len, d_ext, n_fgrams, d_flags, n_entries, s, &flags);
  } while (0);
  if (rc != SCONE_OK) cudaStreamSynchronize(s);   // copies may still read the host vectors
  if (d_tok) cudaFree(d_tok);
  if (d_len) cudaFree(d_len);
  if (d_ext) cudaFree(d_ext);
  if (d_flags) cudaFree(d_flags);
  if (rc != SCONE_OK) {
    cudaGetLastError();
    scone_table_destroy(t);
    return rc;
  }
  in.max_insert_probe = flags.max_kicks;
  *out = t;
  return SCONE_OK;
}

extern "C" int scone_table_destroy(scone_table* t) {
  if (!t) return SCONE_OK;
  int prev = -1;
  cudaGetDevice(&prev);
  if (prev != t->device) cudaSetDevice(t->device);
  if (t->slots || t->status || t->zero_row) cudaDeviceSynchronize();
  if (t->prescan) prescan_release(t->prescan);
  if (t->slots) cudaFree(t->slots);
  if (t->status) cudaFree(t->status);
  if (t->status_host) cudaFreeHost(t->status_host);
  if (t->zero_row) cudaFree(t->zero_row);
  if (prev >= 0 && prev != t->device) cudaSetDevice(prev);
  delete t;
  return SCONE_OK;
}

extern "C" int scone_table_get_info(const scone_table* t, scone_table_info* info) {
  if (!t || !info) return SCONE_ERR_INVALID_ARG;
  *info = t->info;
  return SCONE_OK;
}

extern "C" int scone_table_set_probe_limit(scone_table* t, int64_t max_buckets) {
  if (!t || max_buckets < 1) return SCONE_ERR_INVALID_ARG;
  t->view.probe_limit = max_buckets >= 2 ? 2 : 1;
  return SCONE_OK;
}

extern "C" int scone_table_set_copy_mode(scone_table* t, int32_t mode) {
  if (!t || mode < SCONE_COPY_AUTO || mode > SCONE_COPY_PIPELINED) return SCONE_ERR_INVALID_ARG;
  t->copy_mode = mode;
  return SCONE_OK;
}

namespace scone {
namespace {

// Moves the sticky status word into a host-mapped word and clears it, in
// stream order: one launch instead of a copy and a memset.
__global__ void status_fetch_kernel(int* status, int* host_word) {
  *host_word = atomicExch(status, 0);
}

}  // namespace
}  // namespace scone

extern "C" int scone_status(const scone_table* t, void* stream) {
  if (!t) return SCONE_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  if (t->status_host) {
    // the kernel that records an error (the one whose compare-and-swap sets
    // the status word) also writes it to mirror word 0, so after the sync a
    // zero there means no error and nothing is launched. Otherwise word 0 is
    // cleared first (while the status word is set, no kernel writes it) and
    // one kernel moves the status word into word 1 and clears it; an error
    // recorded after that exchange sets word 0 again for the next call.
    if (cudaStreamSynchronize(s) != cudaSuccess) {
      cudaGetLastError();
      return SCONE_ERR_CUDA;
    }
    volatile int* m = t->status_host;
    if (m[0] == 0) return SCONE_OK;
    m[0] = 0;
    scone::status_fetch_kernel<<<1, 1, 0, s>>>(t->status, t->status_host_dev + 1);
    if (cudaGetLastError() != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess) {
      cudaGetLastError();
      return SCONE_ERR_CUDA;
    }
    return m[1];
  }
  int code = 0;
  if (cudaMemcpyAsync(&code, t->status, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaMemsetAsync(t->status, 0, sizeof(int), s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess) {
    cudaGetLastError();
    return SCONE_ERR_CUDA;
  }
  return code;
}

// ------------------------------------------------------------------------
// Host memory for an offloaded F.
//
// The offloaded tier reads scattered rows of F over the host link. Over tens
// of GB, GPU address translation of host pages, not the link, limits random
// row reads: on GB300 (64 KB base pages) random 4 KB rows over 82 GB of
// cudaHostAlloc memory read at about a third of the link's sequential rate,
// and at twice that when the same memory is backed by transparent huge pages.
// So the buffer is an anonymous mapping aligned to the huge-page size,
// advised MADV_HUGEPAGE, touched in parallel, then pinned and mapped with
// cudaHostRegister; if any step fails it falls back to cudaHostAlloc.

namespace scone {
namespace {

struct HostMapping {
  void* base;   // what mmap returned
  size_t len;   // what was mapped
};

std::mutex g_host_mu;
std::map<void*, HostMapping> g_host_maps;   // registered buffers by user address

size_t huge_page_bytes() {
  size_t h = 2u << 20;
  if (FILE* f = std::fopen("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size", "r")) {
    unsigned long long v = 0;
    if (std::fscanf(f, "%llu", &v) == 1 && v >= 4096 && (v & (v - 1)) == 0) h = (size_t)v;
    std::fclose(f);
  }
  return h;
}

void* map_huge(size_t bytes, HostMapping* m) {
  const size_t huge = huge_page_bytes();
  const size_t plen = (bytes + huge - 1) / huge * huge;
  const size_t len = plen + huge;
  void* base = mmap(nullptr, len, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (base == MAP_FAILED) return nullptr;
  uint8_t* p = reinterpret_cast<uint8_t*>(((uintptr_t)base + huge - 1) / huge * huge);
  madvise(p, plen, MADV_HUGEPAGE);
  // first touch, one write per base page, spread over the host cores
  const size_t page = (size_t)sysconf(_SC_PAGESIZE) > 0 ? (size_t)sysconf(_SC_PAGESIZE) : 4096;
  unsigned nt = std::thread::hardware_concurrency();
  nt = nt < 1 ? 1 : (nt > 32 ? 32 : nt);
  const size_t chunk = (plen / nt + huge - 1) / huge * huge;
  std::vector<std::thread> pool;
  for (unsigned t = 0; t < nt; ++t) {
    const size_t a = t * chunk, b = a + chunk < plen ? a + chunk : plen;
    if (a >= b) break;
    pool.emplace_back([=] {
      for (size_t o = a; o < b; o += page) p[o] = 0;
    });
  }
  for (auto& th : pool) th.join();
  m->base = base;
  m->len = len;
  return p;
}

}  // namespace
}  // namespace scone

extern "C" int scone_host_alloc(int64_t bytes, void** out) {
  if (!out) return SCONE_ERR_INVALID_ARG;
  *out = nullptr;
  if (bytes < 1) return SCONE_ERR_INVALID_ARG;
  HostMapping m{nullptr, 0};
  if (void* p = map_huge((size_t)bytes, &m)) {
    if (cudaHostRegister(p, (size_t)bytes, cudaHostRegisterMapped | cudaHostRegisterPortable) ==
        cudaSuccess) {
      std::lock_guard<std::mutex> lk(g_host_mu);
      g_host_maps[p] = m;
      *out = p;
      return SCONE_OK;
    }
    cudaGetLastError();
    munmap(m.base, m.len);
  }
  void* p = nullptr;
  if (cudaHostAlloc(&p, (size_t)bytes, cudaHostAllocMapped | cudaHostAllocPortable) !=
          cudaSuccess ||
      !p) {
    cudaGetLastError();
    return SCONE_ERR_NOMEM;
  }
  *out = p;
  return SCONE_OK;
}

extern "C" int scone_host_free(void* p) {
  if (!p) return SCONE_OK;
  cudaDeviceSynchronize();
  HostMapping m{nullptr, 0};
  {
    std::lock_guard<std::mutex> lk(g_host_mu);
    auto it = g_host_maps.find(p);
    if (it != g_host_maps.end()) {
      m = it->second;
      g_host_maps.erase(it);
    }
  }
  if (m.base) {
    const bool ok = cudaHostUnregister(p) == cudaSuccess;
    munmap(m.base, m.len);
    return ok ? SCONE_OK : SCONE_ERR_CUDA;
  }
  return cudaFreeHost(p) == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}

extern "C" const char* scone_strerror(int code) {
  switch (code) {
    case SCONE_OK: return "ok";
    case SCONE_ERR_INVALID_ARG: return "invalid argument";
    case SCONE_ERR_TOKEN_RANGE: return "token id outside [0, vocab)";
    case SCONE_ERR_DUPLICATE_FGRAM: return "duplicate f-gram in the list";
    case SCONE_ERR_TABLE_FULL: return "hash table full";
    case SCONE_ERR_PROBE_LIMIT: return "lookup exceeded the probe limit";
    case SCONE_ERR_UNSUPPORTED:
      return "unsupported by this call (key wider than 220 bits, a size past the call's limit, "
             "or a copy mode it cannot use)";
    case SCONE_ERR_CUDA: return "CUDA runtime error";
    case SCONE_ERR_NOMEM: return "out of memory";
    default: return "unknown error";
  }
}

extern "C" int scone_version(void) { return (1 << 16) | 0; }

// ------------------------------------------------------------------------
// Rebuild without allocating (scone_table_rebuild_noalloc).
//
// For callers that cannot allocate when they swap in a new f-gram list: the
// table's slot array, status word and zero row are reused as they are, and
// the build kernels' per-call scratch (device copy of the list, build
// flags) lives in the file-scope array below instead of cudaMalloc'd
// buffers. Host code never uses the array's name as an address: the device
// address is looked up with cudaGetSymbolAddress once per device, with that
// device current, on the first call there.

static __device__ __align__(256) uint8_t g_rebuild_scratch[SCONE_REBUILD_SCRATCH_BYTES];

namespace scone {
namespace {

constexpr int kMaxScratchDevices = 64;
std::mutex g_scratch_mu;
uint8_t* g_scratch_addr[kMaxScratchDevices];  // zero-initialized: not looked up yet

int rebuild_scratch(int dev, uint8_t** out) {
  if (dev < 0 || dev >= kMaxScratchDevices) return SCONE_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_rebuild_scratch) != cudaSuccess || !p) {
      cudaGetLastError();
      return SCONE_ERR_CUDA;
    }
    g_scratch_addr[dev] = static_cast<uint8_t*>(p);
  }
  *out = g_scratch_addr[dev];
  return SCONE_OK;
}

constexpr int64_t round256(int64_t x) { return (x + 255) / 256 * 256; }

}  // namespace
}  // namespace scone

extern "C" int scone_table_rebuild_noalloc(scone_table* t, const int32_t* fgram_tok,
                                           const uint8_t* fgram_len, int64_t n_fgrams,
                                           const scone_bf16* F, void* stream) {
  if (!t || n_fgrams < 0) return SCONE_ERR_INVALID_ARG;
  if (n_fgrams > 0 && (!fgram_tok || !fgram_len || !F)) return SCONE_ERR_INVALID_ARG;
  const int K = t->view.K, vocab = t->view.vocab, d = t->view.d;
  // the new list must fit the existing slot array at load factor <= 0.85
  if ((double)n_fgrams > 0.85 * (double)t->info.n_slots) return SCONE_ERR_INVALID_ARG;
  // scratch layout: [flags: 64 B][fgram_len: n B][fgram_tok: n * K * 4 B], 256-aligned parts
  const int64_t off_len = 256;
  const int64_t off_tok = off_len + round256(n_fgrams);
  const int64_t need = off_tok + round256(n_fgrams * K * 4);
  if (n_fgrams > 0 && need > (int64_t)SCONE_REBUILD_SCRATCH_BYTES) return SCONE_ERR_INVALID_ARG;
  for (int64_t r = 0; r < n_fgrams; ++r) {
    const int n = fgram_len[r];
    if (n < 2 || n > K) return SCONE_ERR_INVALID_ARG;
    for (int j = 0; j < n; ++j)
      if (fgram_tok[r * K + j] < 0 || fgram_tok[r * K + j] >= vocab) return SCONE_ERR_INVALID_ARG;
  }
  DeviceGuard g(t->device);
  const uint16_t* F_dev = reinterpret_cast<const uint16_t*>(F);
  if (n_fgrams > 0) {
    if (t->info.F_location == SCONE_ROWS_DEVICE) {
      if (!is_device_accessible(F)) return SCONE_ERR_INVALID_ARG;
    } else {
      void* dp = nullptr;
      if (cudaHostGetDevicePointer(&dp, const_cast<scone_bf16*>(F), 0) != cudaSuccess || !dp) {
        cudaGetLastError();
        return SCONE_ERR_INVALID_ARG;
      }
      F_dev = reinterpret_cast<const uint16_t*>(dp);
    }
  }
  uint8_t* scratch = nullptr;
  int rc = rebuild_scratch(t->device, &scratch);
  if (rc != SCONE_OK) return rc;
  BuildFlags* d_flags = reinterpret_cast<BuildFlags*>(scratch);
  uint8_t* d_len = scratch + off_len;
  int32_t* d_tok = reinterpret_cast<int32_t*>(scratch + off_tok);
  cudaStream_t s = (cudaStream_t)stream;
  BuildFlags flags = {0, 0, 0};
  if (cudaMemsetAsync(t->status, 0, sizeof(int), s) != cudaSuccess) {
    cudaGetLastError();
    return SCONE_ERR_CUDA;
  }
  if (n_fgrams > 0) {
    if (cudaMemcpyAsync(d_tok, fgram_tok, (size_t)n_fgrams * K * sizeof(int32_t),
                        cudaMemcpyHostToDevice, s) != cudaSuccess ||
        cudaMemcpyAsync(d_len, fgram_len, (size_t)n_fgrams, cudaMemcpyHostToDevice, s) !=
            cudaSuccess) {
      cudaGetLastError();
      return SCONE_ERR_CUDA;
    }
  }
  // the array keeps the previous call's contents: build_slots clears the
  // flags (which must start at zero) before every attempt. The rebuilt
  // slots carry no suffix index (computing one needs host memory): from here
  // on launches take every length independently.
  t->view.suffix_index = 0;
  t->info.n_markers = 0;
  t->info.suffix_index = 0;
  rc = build_slots(t, d_tok, d_len, nullptr, n_fgrams, d_flags, n_fgrams, s, &flags);
  if (rc == SCONE_ERR_CUDA) {
    // the slot array may hold part of the new list while view.F, n_fgrams and
    // the hash seed still describe the old one: one best-effort attempt to
    // leave the table empty (every position falls back to T), as the other
    // failure paths do. If even that fails the table must be destroyed.
    cudaGetLastError();
    if (cudaMemsetAsync(t->slots, 0xFF, (size_t)t->info.table_bytes, s) == cudaSuccess &&
        cudaStreamSynchronize(s) == cudaSuccess) {
      t->view.n_fgrams = 0;
      t->info.n_fgrams = 0;
      t->info.max_insert_probe = 0;
      t->info.F_bytes = 0;
    }
    cudaGetLastError();
    return rc;
  }
  if (rc != SCONE_OK) {
    // leave a valid, empty table: every position falls back to T
    if (cudaMemsetAsync(t->slots, 0xFF, (size_t)t->info.table_bytes, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess) {
      cudaGetLastError();
      return SCONE_ERR_CUDA;
    }
    n_fgrams = 0;
    flags.max_kicks = 0;
  }
  t->view.n_fgrams = n_fgrams;
  t->view.F = n_fgrams > 0 ? F_dev : t->view.F;
  t->info.n_fgrams = n_fgrams;
  t->info.max_insert_probe = flags.max_kicks;
  t->info.F_bytes = n_fgrams * (int64_t)d * 2;
  return rc;
}
