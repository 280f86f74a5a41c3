// Decode step: one new token per live sequence (Sec. 3.2: at inference F is
// looked up per generated token while T stays on the accelerator).
//
// Algorithm 1 only needs the last K-1 tokens before a position, so the state
// keeps, per sequence, a device ring of its last K-1 tokens (right-aligned,
// oldest first) and how many of them are known. One warp serves one
// sequence: lane j looks up the window of length j + 2 ending at the new
// token, a warp ballot keeps the longest hit, the lanes shift the new token
// into the history, and the warp copies the selected row (F over the host
// link in the offloaded tier, or T from HBM) with every lane's loads issued
// at once.
//
// A step is a chain of dependent reads, so its reads are issued as early as
// their addresses are known: the new token, the history length and the
// history entries in one round trip (lane j reads entry j and the window
// tokens reach the other lanes by shuffles), then both candidate buckets of
// every length in one round trip (a second 32-byte sector per lookup instead
// of a second dependent read), then the row.
//
// Steps are launched with programmatic dependent launch: each step lets the
// next one be scheduled at once (griddepcontrol.launch_dependents) and every
// step waits on the device (griddepcontrol.wait) until the previous grid has
// completed and its writes (the history ring) are visible. The launch
// latency between consecutive steps overlaps the running step; the data
// dependency is kept in full. Without a preceding programmatic launch the
// wait returns at once.

#include <new>

#include "scone_host.h"
#include "scone_ptx.cuh"

namespace scone {

constexpr int kDecThreads = 128;
constexpr int kDecWarps = kDecThreads / 32;
constexpr uint32_t kDecSpinLimit = 1u << 22;
constexpr int kDecBulkMaxSmem = 192 * 1024;   // rows of a block's warps staged for bulk copies

namespace {

// W: row copy width (16 or 0 = generic) for register copies. BULK: with
// SCONE_COPY_BULK the selected row moves by TMA bulk copies instead: lane 0
// copies it host/global -> shared (one cp.async.bulk, completion counted in
// bytes on the warp's mbarrier) -> output (cp.async.bulk store), so a row is
// one DMA request per direction and holds no registers. Every wait is
// bounded: past kDecSpinLimit polls the warp records SCONE_ERR_CUDA and
// stops copying.
template <int FMT, int W, bool BULK>
__global__ void __launch_bounds__(kDecThreads)
    decode_kernel(const TableView t, int32_t* __restrict__ hist, int32_t* __restrict__ hist_len,
                  const int32_t* __restrict__ new_tok, int32_t S, int32_t H,
                  uint8_t* __restrict__ out, int32_t* __restrict__ row_out,
                  uint8_t* __restrict__ len_out, int width, const uint8_t* __restrict__ zero_row) {
  constexpr int NW = Fmt<FMT>::kWords;
  __shared__ const void* src_s[kDecWarps][1];
  __shared__ __align__(8) uint64_t bulk_bar[kDecWarps];
  extern __shared__ __align__(128) uint8_t dec_rows[];   // [kDecWarps][row_bytes] (BULK)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int row_bytes = t.d * 2;
  if (BULK && threadIdx.x == 0) {
    for (int w = 0; w < kDecWarps; ++w) mbar_init(saddr(&bulk_bar[w]), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (BULK) __syncthreads();
  uint32_t phase = 0;
  bool broken = false;
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;");
  for (int64_t s = (int64_t)blockIdx.x * kDecWarps + warp; s < S;
       s += (int64_t)gridDim.x * kDecWarps) {
    int32_t* hs = hist + s * H;
    // one round trip: the new token, the history length, history entry `lane`
    const int32_t x = __ldg(new_tok + s);
    const int32_t h = hist_len[s];
    const int32_t hv = lane < H ? hs[lane] : 0;
    const bool xvalid = valid_token(x, t.vocab);
    const int n = lane + 2;
    int32_t r_lane = -1;
    int err = 0;
    KeyBits<NW> k;
#pragma unroll
    for (int q = 0; q < NW; ++q) k.w[q] = 0;
    k.w[0] = (uint32_t)x;
    bool ok = true;
    for (int m = 1; m < H + 1; ++m) {     // every lane joins each shuffle
      const int32_t y = __shfl_sync(0xFFFFFFFFu, hv, H - m);
      if (m < n) {
        ok = ok && valid_token(y, t.vocab);
        put_field<NW>(k, m * t.bits, (uint32_t)y, t.bits);
      }
    }
    if (xvalid && ok && n <= t.K && n <= h + 1) {
      put_len<FMT>(k, n);
      r_lane = cuckoo_lookup_eager<FMT>(t, k, &err);
    }
    const unsigned hits = __ballot_sync(0xFFFFFFFFu, r_lane >= 0);
    const unsigned errs = __ballot_sync(0xFFFFFFFFu, err != 0);
    const int best = hits ? 31 - __clz(hits) : -1;
    int32_t r = __shfl_sync(0xFFFFFFFFu, r_lane, best >= 0 ? best : 0);
    // a probe-limit error matters only at a length longer than the best hit,
    // the same outcome as the longest-first scan of the prefill path
    const bool probe_err = (best >= 0 ? (errs >> (best + 1)) : errs) != 0;
    int len;
    const void* src = nullptr;
    if (!xvalid || probe_err) {
      r = -1;
      len = 0;
    } else {
      if (best < 0) r = -1;
      len = best >= 0 ? best + 2 : 1;
      src = r >= 0 ? static_cast<const void*>(t.F + (int64_t)r * t.d)
                   : static_cast<const void*>(t.T + (int64_t)x * t.d);
    }
    // shift the new token into the history (entry j takes entry j + 1)
    const int32_t next = __shfl_down_sync(0xFFFFFFFFu, hv, 1);
    if (lane < H) hs[lane] = lane + 1 < H ? next : x;
    if (lane == 0) {
      hist_len[s] = h + 1 < H ? h + 1 : H;
      if (row_out) row_out[s] = r;
      if (len_out) len_out[s] = (uint8_t)len;
      if (!xvalid) record_error(t, SCONE_ERR_TOKEN_RANGE);
      else if (probe_err) record_error(t, SCONE_ERR_PROBE_LIMIT);
      src_s[warp][0] = src;
    }
    __syncwarp();
    if (out) {   // NULL: selection only (the rows are gathered elsewhere, e.g. from a row store)
      if constexpr (BULK) {
        if (lane == 0 && !broken) {
          const void* from = src_s[warp][0] ? src_s[warp][0] : (const void*)zero_row;
          uint8_t* buf = dec_rows + warp * row_bytes;
          const uint32_t bar = saddr(&bulk_bar[warp]);
          bulk_wait_read_all();   // this warp's previous row store has read the buffer
          mbar_expect_tx(bar, (uint32_t)row_bytes);
          bulk_load(saddr(buf), from, (uint32_t)row_bytes, bar);
          if (mbar_wait_bounded(bar, phase, kDecSpinLimit)) {
            bulk_store(out + s * (int64_t)row_bytes, saddr(buf), (uint32_t)row_bytes);
            bulk_commit();
            phase ^= 1;
          } else {
            record_error(t, SCONE_ERR_CUDA);
            broken = true;
          }
        }
      } else {
        warp_copy_rows_w<W>(src_s[warp], out + s * (int64_t)row_bytes, 1, row_bytes, width,
                            lane);
      }
    }
    __syncwarp();
  }
  if constexpr (BULK) {
    if (lane == 0) {
      if (broken) mbar_wait_bounded(saddr(&bulk_bar[warp]), phase, kDecSpinLimit);
      bulk_wait_all();   // the row stores complete before the grid does
    }
  }
}

using DecodeFn = void (*)(TableView, int32_t*, int32_t*, const int32_t*, int32_t, int32_t,
                          uint8_t*, int32_t*, uint8_t*, int, const uint8_t*);

DecodeFn pick_decode(int fmt, int width, bool bulk) {
  if (bulk) return fmt == FMT16 ? decode_kernel<FMT16, 16, true> : decode_kernel<FMT32, 16, true>;
  if (fmt == FMT16)
    return width == 16 ? decode_kernel<FMT16, 16, false> : decode_kernel<FMT16, 0, false>;
  return width == 16 ? decode_kernel<FMT32, 16, false> : decode_kernel<FMT32, 0, false>;
}

// Bulk row copies need 16-byte rows and addresses and room for a row per warp.
bool decode_bulk_ok(const scone_table* tb, const void* out) {
  const TableView& t = tb->view;
  const int64_t row_bytes = (int64_t)t.d * 2;
  if (tb->copy_mode != SCONE_COPY_BULK || !out || !tb->zero_row) return false;
  if (row_bytes % 16 || row_bytes * kDecWarps > kDecBulkMaxSmem) return false;
  uintptr_t a = (uintptr_t)t.T | (uintptr_t)out | (uintptr_t)tb->zero_row;
  if (t.n_fgrams > 0) a |= (uintptr_t)t.F;
  return (a & 15) == 0;
}

}  // namespace

}  // namespace scone

using namespace scone;

extern "C" int scone_decode_create(const scone_table* tb, int32_t S, const int32_t* hist,
                                   const int32_t* hist_len, scone_decode** out) {
  if (!out) return SCONE_ERR_INVALID_ARG;
  *out = nullptr;
  if (!tb || S < 0 || (S > 0 && (!hist || !hist_len))) return SCONE_ERR_INVALID_ARG;
  const int32_t H = tb->view.K - 1;
  for (int32_t s = 0; s < S; ++s)
    if (hist_len[s] < 0 || hist_len[s] > H) return SCONE_ERR_INVALID_ARG;
  DeviceGuard g(tb->device);
  scone_decode* st = new (std::nothrow) scone_decode();
  if (!st) return SCONE_ERR_NOMEM;
  st->table = tb;
  st->S = S;
  st->H = H;
  if (S > 0) {
    if (cudaMalloc(&st->hist, (size_t)S * H * sizeof(int32_t)) != cudaSuccess ||
        cudaMalloc(&st->hist_len, (size_t)S * sizeof(int32_t)) != cudaSuccess) {
      cudaGetLastError();
      scone_decode_destroy(st);
      return SCONE_ERR_NOMEM;
    }
    if (cudaMemcpy(st->hist, hist, (size_t)S * H * sizeof(int32_t), cudaMemcpyHostToDevice) !=
            cudaSuccess ||
        cudaMemcpy(st->hist_len, hist_len, (size_t)S * sizeof(int32_t),
                   cudaMemcpyHostToDevice) != cudaSuccess) {
      cudaGetLastError();
      scone_decode_destroy(st);
      return SCONE_ERR_CUDA;
    }
  }
  *out = st;
  return SCONE_OK;
}

extern "C" int scone_decode_step(scone_decode* st, const int32_t* new_tok, scone_bf16* out,
                                 int32_t* row, uint8_t* len, void* stream) {
  if (!st || !st->table) return SCONE_ERR_INVALID_ARG;
  if (st->S == 0) return SCONE_OK;
  if (!new_tok || (!out && !row) || ((uintptr_t)new_tok & 3) || ((uintptr_t)out & 1) ||
      (row && ((uintptr_t)row & 3)))
    return SCONE_ERR_INVALID_ARG;
  const scone_table* tb = st->table;
  DeviceGuard g(tb->device);
  const int width = row_copy_width(tb->view, out);
  const bool bulk = decode_bulk_ok(tb, out);
  const DecodeFn fn = pick_decode(tb->fmt, width, bulk);
  const size_t smem = bulk ? (size_t)kDecWarps * tb->view.d * 2 : 0;
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute((const void*)fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem) != cudaSuccess) {
    cudaGetLastError();
    return SCONE_ERR_CUDA;
  }
  const int64_t need = (st->S + kDecWarps - 1) / kDecWarps;
  const int64_t cap = (int64_t)sm_count() * blocks_per_sm((const void*)fn, kDecThreads, smem);
  const int grid = (int)(need < cap ? need : cap);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kDecThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = (cudaStream_t)stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, fn, tb->view, st->hist, st->hist_len, new_tok,
                                           st->S, st->H, reinterpret_cast<uint8_t*>(out), row,
                                           len, width, (const uint8_t*)tb->zero_row);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return SCONE_ERR_CUDA;
  }
  return SCONE_OK;
}

extern "C" int scone_decode_get_history(const scone_decode* st, int32_t* hist,
                                        int32_t* hist_len) {
  if (!st || (st->S > 0 && (!hist || !hist_len))) return SCONE_ERR_INVALID_ARG;
  if (st->S == 0) return SCONE_OK;
  DeviceGuard g(st->table->device);
  if (cudaDeviceSynchronize() != cudaSuccess ||
      cudaMemcpy(hist, st->hist, (size_t)st->S * st->H * sizeof(int32_t),
                 cudaMemcpyDeviceToHost) != cudaSuccess ||
      cudaMemcpy(hist_len, st->hist_len, (size_t)st->S * sizeof(int32_t),
                 cudaMemcpyDeviceToHost) != cudaSuccess) {
    cudaGetLastError();
    return SCONE_ERR_CUDA;
  }
  return SCONE_OK;
}

extern "C" int scone_decode_destroy(scone_decode* st) {
  if (!st) return SCONE_OK;
  if (st->hist || st->hist_len) {
    DeviceGuard g(st->table ? st->table->device : 0);
    cudaDeviceSynchronize();
    if (st->hist) cudaFree(st->hist);
    if (st->hist_len) cudaFree(st->hist_len);
  }
  delete st;
  return SCONE_OK;
}
