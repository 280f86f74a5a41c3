// Row store: F kept in a file, beyond host memory (the paper's storage tier,
// Sec. 4.3: the f-gram embeddings on solid-state drives, read per token).
//
// The file holds F row after row (n_rows x d bf16, no header). The store
// keeps a direct-mapped cache of rows in HBM (cache_rows slots, slot =
// mix(row) mod cache_rows, a row-id tag per slot). One gather call:
//   1. lookup_kernel: every position copies its row from the cache (a hit),
//      from T (the token fallback), or records a miss (position, row);
//   2. the host reads the misses' distinct rows from the file with pread
//      (O_DIRECT when rows are 4 KiB multiples, so the page cache is not the
//      tier) on a pool of threads into pinned staging, and picks the cache
//      slots to fill (the first missed row of each slot in the call);
//   3. fill_kernel copies the staged rows to the missed positions and into
//      their cache slots, updating the tags.
// Hot rows of a Zipf workload stay in HBM; cold rows cost one file read.

#include <fcntl.h>
#include <sys/stat.h>
#include <unistd.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <cstdlib>
#include <condition_variable>
#include <cstring>
#include <functional>
#include <mutex>
#include <new>
#include <thread>
#include <unordered_map>
#include <vector>

#include "scone_host.h"

namespace scone {
namespace {

constexpr int kStoreThreads = 256;
constexpr int kStoreWarps = kStoreThreads / 32;

__device__ __forceinline__ uint64_t slot_of_row(int64_t r, int64_t cache_rows) {
  return fmix64((uint64_t)r ^ 0x3C6EF372FE94F82Bull) % (uint64_t)cache_rows;
}
uint64_t host_fmix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
uint64_t host_slot_of_row(int64_t r, int64_t cache_rows) {
  return host_fmix64((uint64_t)r ^ 0x3C6EF372FE94F82Bull) % (uint64_t)cache_rows;
}

// Step 1: one warp per 32 positions; lanes choose sources, the warp copies.
__global__ void __launch_bounds__(kStoreThreads)
    lookup_kernel(const TableView t, const int32_t* __restrict__ tok,
                  const int32_t* __restrict__ row, int64_t n, const uint16_t* __restrict__ cache,
                  const int64_t* __restrict__ tag, int64_t cache_rows, int64_t n_rows,
                  uint8_t* __restrict__ out, int32_t* __restrict__ miss_pos,
                  int32_t* __restrict__ miss_row, int* __restrict__ miss_count, int width) {
  __shared__ const void* src_s[kStoreWarps][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int row_bytes = t.d * 2;
  const int64_t stride = (int64_t)gridDim.x * kStoreThreads;
  for (int64_t base = ((int64_t)blockIdx.x * kStoreWarps + warp) * 32; base < n;
       base += stride) {
    const int nrows = (int)(n - base < 32 ? n - base : 32);
    const int64_t p = base + lane;
    const void* src = nullptr;
    if (lane < nrows) {
      const int32_t r = row[p];
      if (r < 0) {
        const int32_t x = tok[p];
        if (valid_token(x, t.vocab)) src = t.T + (int64_t)x * t.d;
        else record_error(t, SCONE_ERR_TOKEN_RANGE);
      } else if (r >= n_rows) {
        record_error(t, SCONE_ERR_INVALID_ARG);
      } else {
        const uint64_t s = slot_of_row(r, cache_rows);
        if (tag[s] == r) {
          src = cache + s * (int64_t)t.d;
        } else {
          const int k = atomicAdd(miss_count, 1);
          miss_pos[k] = (int32_t)p;
          miss_row[k] = r;
        }
      }
    }
    src_s[warp][lane] = src;
    __syncwarp();
    if (width == 16)
      warp_copy_rows_w<16>(src_s[warp], out + base * (int64_t)row_bytes, nrows, row_bytes, 16,
                           lane);
    else
      warp_copy_rows_w<0>(src_s[warp], out + base * (int64_t)row_bytes, nrows, row_bytes, width,
                          lane);
    __syncwarp();
  }
}

// Step 3: one warp per missed position (its staged row to out), then one
// warp per filled cache slot (its staged row and tag).
__global__ void __launch_bounds__(kStoreThreads)
    fill_kernel(const uint8_t* __restrict__ staged, int64_t row_bytes,
                const int32_t* __restrict__ miss_pos, const int32_t* __restrict__ miss_src,
                int n_miss, const int64_t* __restrict__ fill_slot,
                const int64_t* __restrict__ fill_row, const int32_t* __restrict__ fill_src,
                int n_fill, uint8_t* __restrict__ out, uint8_t* __restrict__ cache,
                int64_t* __restrict__ tag) {
  const int lane = threadIdx.x & 31;
  const int64_t w = (int64_t)blockIdx.x * kStoreWarps + (threadIdx.x >> 5);
  const int64_t n16 = row_bytes / 16;
  if (w < n_miss) {
    const uint4* src = reinterpret_cast<const uint4*>(staged + (int64_t)miss_src[w] * row_bytes);
    uint4* dst = reinterpret_cast<uint4*>(out + (int64_t)miss_pos[w] * row_bytes);
    for (int64_t c = lane; c < n16; c += 32) dst[c] = src[c];
  } else if (w < (int64_t)n_miss + n_fill) {
    const int64_t f = w - n_miss;
    const uint4* src = reinterpret_cast<const uint4*>(staged + (int64_t)fill_src[f] * row_bytes);
    uint4* dst = reinterpret_cast<uint4*>(cache + fill_slot[f] * row_bytes);
    for (int64_t c = lane; c < n16; c += 32) dst[c] = src[c];
    if (lane == 0) tag[fill_slot[f]] = fill_row[f];
  }
}

// A fixed pool of reader threads.
class ReadPool {
 public:
  explicit ReadPool(int n) {
    for (int i = 0; i < n; ++i) workers_.emplace_back([this] { loop(); });
  }
  ~ReadPool() {
    {
      std::lock_guard<std::mutex> lk(mu_);
      stop_ = true;
    }
    cv_.notify_all();
    for (auto& t : workers_) t.join();
  }
  // Runs fn(i) for i in [0, n) on the pool; returns when all are done.
  void run(int64_t n, const std::function<void(int64_t)>& fn) {
    std::atomic<int64_t> next(0);
    std::atomic<int> busy((int)workers_.size());
    {
      std::lock_guard<std::mutex> lk(mu_);
      job_ = [&] {
        for (int64_t i = next++; i < n; i = next++) fn(i);
      };
      pending_ = &busy;
      ++gen_;
    }
    cv_.notify_all();
    std::unique_lock<std::mutex> lk(mu_);
    done_cv_.wait(lk, [&] { return busy.load() == 0; });
    job_ = nullptr;
    pending_ = nullptr;
  }

 private:
  void loop() {
    uint64_t seen = 0;
    for (;;) {
      std::function<void()> job;
      std::atomic<int>* pending;
      {
        std::unique_lock<std::mutex> lk(mu_);
        cv_.wait(lk, [&] { return stop_ || gen_ != seen; });
        if (stop_) return;
        seen = gen_;
        job = job_;
        pending = pending_;
      }
      job();
      if (pending->fetch_sub(1) == 1) {
        std::lock_guard<std::mutex> lk(mu_);
        done_cv_.notify_all();
      }
    }
  }
  std::vector<std::thread> workers_;
  std::mutex mu_;
  std::condition_variable cv_, done_cv_;
  std::function<void()> job_;
  std::atomic<int>* pending_ = nullptr;
  uint64_t gen_ = 0;
  bool stop_ = false;
};

}  // namespace
}  // namespace scone

struct scone_rowstore {
  int device = 0;
  int fd = -1;
  bool direct = false;
  int64_t n_rows = 0;
  int32_t d = 0;
  int64_t row_bytes = 0;
  int64_t cache_rows = 0;
  uint16_t* cache = nullptr;           // device [cache_rows x d]
  int64_t* tag = nullptr;              // device [cache_rows], -1 empty
  // per-call buffers, grown on demand
  int64_t cap = 0;                     // positions
  int32_t *d_miss_pos = nullptr, *d_miss_row = nullptr, *d_miss_src = nullptr;
  int* d_miss_count = nullptr;
  int* h_miss_count = nullptr;         // pinned
  int32_t *h_miss_row = nullptr, *h_miss_src = nullptr;
  int64_t stage_cap = 0;               // staged rows
  uint8_t* h_stage = nullptr;          // pinned, 4096-aligned
  uint8_t* d_stage = nullptr;
  int64_t *h_fill = nullptr, *d_fill = nullptr;   // [2 * stage_cap]: cache slot, row
  int32_t *h_fill_src = nullptr, *d_fill_src = nullptr;   // [stage_cap]: staged index
  scone::ReadPool* pool = nullptr;
  scone_rowstore_stats stats{};
};

namespace scone {
namespace {

void free_call_buffers(scone_rowstore* st) {
  for (void* p : {(void*)st->d_miss_pos, (void*)st->d_miss_row, (void*)st->d_miss_src,
                  (void*)st->d_miss_count, (void*)st->d_stage, (void*)st->d_fill,
                  (void*)st->d_fill_src})
    if (p) cudaFree(p);
  for (void* p : {(void*)st->h_miss_count, (void*)st->h_miss_row, (void*)st->h_miss_src,
                  (void*)st->h_stage, (void*)st->h_fill, (void*)st->h_fill_src})
    if (p) cudaFreeHost(p);
  st->h_miss_count = nullptr;
  st->d_fill_src = st->h_fill_src = nullptr;
  st->d_miss_pos = st->d_miss_row = st->d_miss_src = nullptr;
  st->d_miss_count = nullptr;
  st->d_stage = nullptr;
  st->d_fill = nullptr;
  st->h_miss_row = st->h_miss_src = nullptr;
  st->h_stage = nullptr;
  st->h_fill = nullptr;
  st->cap = st->stage_cap = 0;
}

bool grow(scone_rowstore* st, int64_t n) {
  if (n <= st->cap) return true;
  free_call_buffers(st);
  const int64_t c = n + n / 4 + 64;
  const size_t rb = (size_t)st->row_bytes;
  if (cudaMalloc(&st->d_miss_pos, c * 4) != cudaSuccess ||
      cudaMalloc(&st->d_miss_row, c * 4) != cudaSuccess ||
      cudaMalloc(&st->d_miss_src, c * 4) != cudaSuccess ||
      cudaMalloc(&st->d_miss_count, sizeof(int)) != cudaSuccess ||
      cudaMalloc(&st->d_stage, c * rb) != cudaSuccess ||
      cudaMalloc(&st->d_fill, 2 * c * sizeof(int64_t)) != cudaSuccess ||
      cudaMalloc(&st->d_fill_src, c * 4) != cudaSuccess ||
      cudaHostAlloc(&st->h_miss_count, sizeof(int), cudaHostAllocDefault) != cudaSuccess ||
      cudaHostAlloc(&st->h_miss_row, c * 4, cudaHostAllocDefault) != cudaSuccess ||
      cudaHostAlloc(&st->h_miss_src, c * 4, cudaHostAllocDefault) != cudaSuccess ||
      cudaHostAlloc(&st->h_stage, c * rb, cudaHostAllocDefault) != cudaSuccess ||
      cudaHostAlloc(&st->h_fill, 2 * c * sizeof(int64_t), cudaHostAllocDefault) != cudaSuccess ||
      cudaHostAlloc(&st->h_fill_src, c * 4, cudaHostAllocDefault) != cudaSuccess) {
    cudaGetLastError();
    free_call_buffers(st);
    return false;
  }
  st->cap = st->stage_cap = c;
  return true;
}

// Reads row r of the file into dst (row_bytes); false on a short read.
bool read_row(const scone_rowstore* st, int64_t r, uint8_t* dst) {
  int64_t done = 0;
  const int64_t off = r * st->row_bytes;
  while (done < st->row_bytes) {
    const ssize_t k = pread(st->fd, dst + done, (size_t)(st->row_bytes - done), off + done);
    if (k <= 0) return false;
    done += k;
  }
  return true;
}

}  // namespace
}  // namespace scone

using namespace scone;

extern "C" int scone_rowstore_open(const char* path, int64_t n_rows, int32_t d, int64_t cache_rows,
                                   int32_t threads, scone_rowstore** out) {
  if (!out) return SCONE_ERR_INVALID_ARG;
  *out = nullptr;
  if (!path || n_rows < 1 || d < 8 || d % 8 || cache_rows < 1 || threads < 0)
    return SCONE_ERR_INVALID_ARG;
  const int64_t row_bytes = (int64_t)d * 2;
  const bool direct = row_bytes % 4096 == 0;
  int fd = open(path, O_RDONLY | (direct ? O_DIRECT : 0));
  if (fd < 0 && direct) fd = open(path, O_RDONLY);    // filesystems without O_DIRECT
  if (fd < 0) return SCONE_ERR_INVALID_ARG;
  struct stat sb;
  if (fstat(fd, &sb) != 0 || sb.st_size < n_rows * row_bytes) {
    close(fd);
    return SCONE_ERR_INVALID_ARG;
  }
  auto* st = new (std::nothrow) scone_rowstore();
  if (!st) {
    close(fd);
    return SCONE_ERR_NOMEM;
  }
  cudaGetDevice(&st->device);
  st->fd = fd;
  st->direct = direct && (fcntl(fd, F_GETFL) & O_DIRECT);
  st->n_rows = n_rows;
  st->d = d;
  st->row_bytes = row_bytes;
  st->cache_rows = cache_rows;
  if (cudaMalloc(&st->cache, (size_t)cache_rows * row_bytes) != cudaSuccess ||
      cudaMalloc(&st->tag, (size_t)cache_rows * sizeof(int64_t)) != cudaSuccess ||
      cudaMemset(st->tag, 0xFF, (size_t)cache_rows * sizeof(int64_t)) != cudaSuccess) {
    cudaGetLastError();
    scone_rowstore_close(st);
    return SCONE_ERR_NOMEM;
  }
  const int nt = threads > 0 ? threads : (int)std::max(1u, std::thread::hardware_concurrency());
  st->pool = new (std::nothrow) ReadPool(nt);
  if (!st->pool) {
    scone_rowstore_close(st);
    return SCONE_ERR_NOMEM;
  }
  *out = st;
  return SCONE_OK;
}

extern "C" int scone_rowstore_close(scone_rowstore* st) {
  if (!st) return SCONE_OK;
  DeviceGuard g(st->device);
  cudaDeviceSynchronize();
  delete st->pool;
  free_call_buffers(st);
  if (st->cache) cudaFree(st->cache);
  if (st->tag) cudaFree(st->tag);
  if (st->fd >= 0) close(st->fd);
  delete st;
  return SCONE_OK;
}

extern "C" int scone_rowstore_get_stats(const scone_rowstore* st, scone_rowstore_stats* out) {
  if (!st || !out) return SCONE_ERR_INVALID_ARG;
  *out = st->stats;
  out->direct_io = st->direct ? 1 : 0;
  return SCONE_OK;
}

extern "C" int scone_rowstore_gather(scone_rowstore* st, const scone_table* tb,
                                     const int32_t* tok, const int32_t* row, int64_t n,
                                     scone_bf16* out, void* stream) {
  if (!st || !tb || n < 0 || n > 0x7FFFFFFF) return SCONE_ERR_INVALID_ARG;
  if (n == 0) return SCONE_OK;
  if (!tok || !row || !out || tb->view.d != st->d || ((uintptr_t)out & 15) ||
      ((uintptr_t)tok & 3) || ((uintptr_t)row & 3))
    return SCONE_ERR_INVALID_ARG;
  DeviceGuard g(st->device);
  cudaStream_t s = (cudaStream_t)stream;
  if (!grow(st, n)) return SCONE_ERR_NOMEM;
  const TableView& t = tb->view;
  const int width = row_copy_width(t, out, (uintptr_t)st->cache);
  const int64_t blocks_needed = (n + kStoreThreads - 1) / kStoreThreads;
  const int64_t cap = (int64_t)sm_count() * blocks_per_sm((const void*)lookup_kernel,
                                                          kStoreThreads, 0);
  const int grid = (int)(blocks_needed < cap ? blocks_needed : cap);
  if (cudaMemsetAsync(st->d_miss_count, 0, sizeof(int), s) != cudaSuccess) return SCONE_ERR_CUDA;
  lookup_kernel<<<grid, kStoreThreads, 0, s>>>(t, tok, row, n, st->cache, st->tag,
                                               st->cache_rows, st->n_rows,
                                               reinterpret_cast<uint8_t*>(out), st->d_miss_pos,
                                               st->d_miss_row, st->d_miss_count, width);
  if (cudaGetLastError() != cudaSuccess ||
      cudaMemcpyAsync(st->h_miss_count, st->d_miss_count, sizeof(int), cudaMemcpyDeviceToHost,
                      s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return SCONE_ERR_CUDA;
  const int n_miss = *st->h_miss_count;
  st->stats.positions += n;
  st->stats.misses += n_miss;
  if (n_miss == 0) return SCONE_OK;
  if (cudaMemcpyAsync(st->h_miss_row, st->d_miss_row, (size_t)n_miss * 4, cudaMemcpyDeviceToHost,
                      s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return SCONE_ERR_CUDA;
  // distinct missed rows, each staged once; the first of each slot fills it
  std::unordered_map<int32_t, int32_t> staged_of;
  staged_of.reserve((size_t)n_miss * 2);
  std::vector<int32_t> uniq;
  for (int k = 0; k < n_miss; ++k) {
    const int32_t r = st->h_miss_row[k];
    auto it = staged_of.find(r);
    if (it == staged_of.end()) {
      it = staged_of.emplace(r, (int32_t)uniq.size()).first;
      uniq.push_back(r);
    }
    st->h_miss_src[k] = it->second;
  }
  const int64_t nu = (int64_t)uniq.size();
  std::atomic<bool> io_ok(true);
  st->pool->run(nu, [&](int64_t u) {
    if (!read_row(st, uniq[(size_t)u], st->h_stage + u * st->row_bytes)) io_ok = false;
  });
  if (!io_ok) return SCONE_ERR_CUDA;
  // cache fills: one per slot, the first distinct missed row that maps to it
  int64_t n_fill = 0;
  int64_t* fill_slot = st->h_fill;
  int64_t* fill_row = st->h_fill + st->stage_cap;
  std::unordered_map<int64_t, char> slot_taken;
  slot_taken.reserve((size_t)nu * 2);
  for (int64_t u = 0; u < nu; ++u) {
    const int64_t slot = (int64_t)host_slot_of_row(uniq[(size_t)u], st->cache_rows);
    if (!slot_taken.emplace(slot, 1).second) continue;
    fill_slot[n_fill] = slot;
    fill_row[n_fill] = uniq[(size_t)u];
    st->h_fill_src[n_fill] = (int32_t)u;
    ++n_fill;
  }
  if (cudaMemcpyAsync(st->d_stage, st->h_stage, (size_t)nu * st->row_bytes,
                      cudaMemcpyHostToDevice, s) != cudaSuccess ||
      cudaMemcpyAsync(st->d_miss_src, st->h_miss_src, (size_t)n_miss * 4, cudaMemcpyHostToDevice,
                      s) != cudaSuccess ||
      cudaMemcpyAsync(st->d_fill, fill_slot, (size_t)n_fill * 8, cudaMemcpyHostToDevice, s) !=
          cudaSuccess ||
      cudaMemcpyAsync(st->d_fill + st->stage_cap, fill_row, (size_t)n_fill * 8,
                      cudaMemcpyHostToDevice, s) != cudaSuccess ||
      cudaMemcpyAsync(st->d_fill_src, st->h_fill_src, (size_t)n_fill * 4,
                      cudaMemcpyHostToDevice, s) != cudaSuccess)
    return SCONE_ERR_CUDA;
  const int64_t warps = (int64_t)n_miss + n_fill;
  fill_kernel<<<(unsigned)((warps + kStoreWarps - 1) / kStoreWarps), kStoreThreads, 0, s>>>(
      st->d_stage, st->row_bytes, st->d_miss_pos, st->d_miss_src, n_miss, st->d_fill,
      st->d_fill + st->stage_cap, st->d_fill_src, (int)n_fill, reinterpret_cast<uint8_t*>(out),
      reinterpret_cast<uint8_t*>(st->cache), st->tag);
  if (cudaGetLastError() != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess)
    return SCONE_ERR_CUDA;
  st->stats.rows_read += nu;
  st->stats.bytes_read += nu * st->row_bytes;
  return SCONE_OK;
}

extern "C" int scone_rowstore_probe_reads(scone_rowstore* st, int64_t n_reads, uint64_t seed,
                                          double* rows_per_s, double* bytes_per_s) {
  if (!st || n_reads < 1 || !rows_per_s || !bytes_per_s) return SCONE_ERR_INVALID_ARG;
  // landing buffers, 4096-aligned for O_DIRECT; contents are discarded, so
  // reads that share a buffer may overlap
  const int64_t n_buf = n_reads < 256 ? n_reads : 256;
  void* buf = nullptr;
  if (posix_memalign(&buf, 4096, (size_t)(n_buf * st->row_bytes)) != 0) return SCONE_ERR_NOMEM;
  std::vector<int64_t> rows((size_t)n_reads);
  for (int64_t i = 0; i < n_reads; ++i)
    rows[(size_t)i] = (int64_t)(host_fmix64(seed + (uint64_t)i * 0x9E3779B97F4A7C15ull) %
                                (uint64_t)st->n_rows);
  std::atomic<bool> io_ok(true);
  const auto t0 = std::chrono::steady_clock::now();
  st->pool->run(n_reads, [&](int64_t i) {
    uint8_t* dst = static_cast<uint8_t*>(buf) + (i % n_buf) * st->row_bytes;
    if (!read_row(st, rows[(size_t)i], dst)) io_ok = false;
  });
  const double sec = std::chrono::duration<double>(std::chrono::steady_clock::now() - t0).count();
  free(buf);
  if (!io_ok) return SCONE_ERR_CUDA;
  *rows_per_s = (double)n_reads / sec;
  *bytes_per_s = (double)n_reads * (double)st->row_bytes / sec;
  return SCONE_OK;
}
