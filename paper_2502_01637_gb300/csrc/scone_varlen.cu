// Ragged and continued batches (Algorithm 1 over packed sequences of any
// lengths, optionally continuing sequences kept in a decode state).
//
// A batch is n_seq sequences packed back to back, sequence b at
// tok[cu[b] .. cu[b+1]). Without a state every sequence starts at its first
// token, as in scone_embed. With a state, sequence b continues state slot
// slot[b]: the last K-1 tokens seen so far in that slot (its history) come
// before the chunk, so the windows of the chunk's first K-1 positions reach
// into the history. That covers chunked prefill (a long prompt in pieces),
// decode (chunks of one token), and batches mixing both in one launch.
//
// varlen_embed_kernel is the fused kernel's scheme (persistent grid, an even
// split of positions over warps, a lane per position, then a warp-wide row
// copy) with two changes per lane: the sequence of position p is found in cu
// (the last b with cu[b] <= p, so empty sequences are skipped) by a galloping
// search that starts at the sequence of the warp's previous tile, and window
// tokens left of the chunk come from the history. varlen_hist_kernel then
// replaces each continued slot's history with the last K-1 tokens of
// history ++ chunk; it is a separate launch because the embedding kernel's
// lanes read the old history, made with programmatic dependent launch: it is
// scheduled while the embedding kernel runs and waits on the device
// (griddepcontrol.wait) until that grid has finished.

#include "scone_host.h"

namespace scone {

namespace {

constexpr int kVThreads = 256;
constexpr int kVWarps = kVThreads / 32;

// Last b in [b0, n_seq) with cu[b] <= p, given cu[b0] <= p (b0 = 0, or the
// sequence of an earlier position): steps of 1, 2, 4, .. from b0 until one
// overshoots, then a binary search below it. A position in the sequence of
// the previous one costs one read; indices stay in [b0, n_seq).
__device__ __forceinline__ int32_t seq_from(const int32_t* __restrict__ cu, int32_t n_seq,
                                            int64_t p, int32_t b0) {
  int32_t lo = b0, hi = n_seq - 1, step = 1;
  while (lo < hi) {
    const int32_t probe = hi - lo > step ? lo + step : hi;
    if ((int64_t)__ldg(cu + probe) <= p) {
      lo = probe;
      step <<= 1;
    } else {
      hi = probe - 1;
      break;
    }
  }
  while (lo < hi) {
    const int32_t mid = (lo + hi + 1) >> 1;
    if ((int64_t)__ldg(cu + mid) <= p) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// Selection for packed position p. Sets *len / *err like match_position; a
// slot outside [0, S) is SCONE_ERR_INVALID_ARG.
template <int FMT, int KT>
__device__ __forceinline__ int32_t match_varlen(const TableView& t,
                                                const int32_t* __restrict__ tok,
                                                const int32_t* __restrict__ cu, int32_t b,
                                                const int32_t* __restrict__ hist,
                                                const int32_t* __restrict__ hist_len,
                                                const int32_t* __restrict__ slot, int32_t S,
                                                int32_t H, int64_t p, int32_t x, int* len,
                                                int* err) {
  if (!valid_token(x, t.vocab)) {
    *err = SCONE_ERR_TOKEN_RANGE;
    *len = 0;
    return -1;
  }
  const int32_t c0 = __ldg(cu + b);
  const int64_t i = p - (c0 > 0 ? c0 : 0);   // offset in the chunk, never left of tok[0]
  int32_t h = 0;
  const int32_t* hrow = nullptr;
  if (hist) {
    const int32_t s = slot ? __ldg(slot + b) : b;
    if (s < 0 || s >= S) {
      *err = SCONE_ERR_INVALID_ARG;
      *len = 0;
      return -1;
    }
    // only the chunk's first K-1 windows reach into the history
    if (i < t.K - 1) h = hist_len[s];
    hrow = hist + (int64_t)s * H;
  }
  const int64_t known = i + 1 + h;        // tokens of the sequence up to p
  const int nmax = known < t.K ? (int)known : t.K;
  const Match m = match_window<FMT, KT>(t, x, nmax, [&](int j) {
    return j <= i ? __ldg(tok + p - j) : hrow[H - (j - i)];
  });
  *len = m.len;
  if (m.err) *err = m.err;
  return m.row;
}

template <int KT>
struct VarlenTuning {
  static constexpr int kLoads = KT <= 3 ? 8 : 16;
  static constexpr int kMinBlocks = KT <= 3 ? 3 : (KT <= 5 ? 2 : 1);
};

template <int FMT, int KT, int W>
__global__ void __launch_bounds__(kVThreads, VarlenTuning<KT>::kMinBlocks)
    varlen_embed_kernel(const TableView t, const int32_t* __restrict__ tok, int64_t n_tok,
                        const int32_t* __restrict__ cu, int32_t n_seq,
                        const int32_t* __restrict__ hist, const int32_t* __restrict__ hist_len,
                        const int32_t* __restrict__ slot, int32_t S, int32_t H,
                        uint8_t* __restrict__ out, int32_t* __restrict__ row_out,
                        uint8_t* __restrict__ len_out, int width) {
  __shared__ const void* src_s[kVWarps][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int row_bytes = t.d * 2;
  // the history kernel that follows may be scheduled now; it waits for this grid
  asm volatile("griddepcontrol.launch_dependents;");
  const int64_t nw = (int64_t)gridDim.x * kVWarps, w = (int64_t)blockIdx.x * kVWarps + warp;
  const int64_t lo = n_tok * w / nw, hi = n_tok * (w + 1) / nw;
  int32_t bq = 0;   // sequence of the warp's previous position (positions only increase)
  for (int64_t base = lo; base < hi; base += 32) {
    const int nrows = (int)(hi - base < 32 ? hi - base : 32);
    const int64_t p = base + lane;
    const void* src = nullptr;
    const int32_t b = lane < nrows ? seq_from(cu, n_seq, p, bq) : bq;
    bq = __shfl_sync(0xFFFFFFFFu, b, nrows - 1);
    if (lane < nrows) {
      const int32_t x = __ldg(tok + p);
      int len = 0, err = 0;
      const int32_t r = match_varlen<FMT, KT>(t, tok, cu, b, hist, hist_len, slot, S, H, p, x,
                                              &len, &err);
      if (err) {
        record_error(t.status, err);
      } else {
        src = r >= 0 ? static_cast<const void*>(t.F + (int64_t)r * t.d)
                     : static_cast<const void*>(t.T + (int64_t)x * t.d);
      }
      if (row_out) row_out[p] = r;
      if (len_out) len_out[p] = (uint8_t)len;
    }
    src_s[warp][lane] = src;
    __syncwarp();
    warp_copy_rows_w<W, VarlenTuning<KT>::kLoads>(src_s[warp], out + base * (int64_t)row_bytes,
                                                  nrows, row_bytes, width, lane);
    __syncwarp();
  }
}

// One thread per sequence: the slot's history becomes the last H tokens of
// history ++ chunk (right-aligned, oldest first), its length min(H, h + c).
__global__ void __launch_bounds__(256)
    varlen_hist_kernel(const int32_t* __restrict__ tok, int64_t n_tok,
                       const int32_t* __restrict__ cu, int32_t n_seq, int32_t* __restrict__ hist,
                       int32_t* __restrict__ hist_len, const int32_t* __restrict__ slot,
                       int32_t S, int32_t H) {
  // launched as a programmatic dependent of the embedding kernel, whose lanes
  // read the histories this kernel rewrites: wait until that grid is done
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int32_t b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= n_seq || H == 0) return;
  const int32_t s = slot ? slot[b] : b;
  if (s < 0 || s >= S) return;          // reported by the embedding kernel
  const int64_t c0 = cu[b], c = (int64_t)cu[b + 1] - c0;
  if (c <= 0 || c0 < 0 || c0 + c > n_tok) return;   // empty, or not a valid chunk
  int32_t* row = hist + (int64_t)s * H;
  const int32_t h = hist_len[s];
  int32_t nw[8];                         // H <= 7
  for (int j = 0; j < H; ++j) {
    // entry j of the new row is the token H - j places from the end of
    // history ++ chunk
    const int64_t back = H - j;          // 1 = the chunk's last token
    nw[j] = back <= c ? tok[c0 + c - back] : row[H - (back - c)];
  }
  for (int j = 0; j < H; ++j) row[j] = nw[j];
  hist_len[s] = (int32_t)(h + c < H ? h + c : H);
}

using VarlenFn = void (*)(TableView, const int32_t*, int64_t, const int32_t*, int32_t,
                          const int32_t*, const int32_t*, const int32_t*, int32_t, int32_t,
                          uint8_t*, int32_t*, uint8_t*, int);

template <int W>
VarlenFn pick_varlen_w(int fmt, int K) {
  if (fmt == FMT16) {
    if (K <= 3) return varlen_embed_kernel<FMT16, 3, W>;
    if (K <= 5) return varlen_embed_kernel<FMT16, 5, W>;
    return varlen_embed_kernel<FMT16, 8, W>;
  }
  if (K <= 5) return varlen_embed_kernel<FMT32, 5, W>;
  return varlen_embed_kernel<FMT32, 8, W>;
}

}  // namespace

}  // namespace scone

using namespace scone;

extern "C" int scone_embed_varlen(const scone_table* tb, const int32_t* tok, int64_t n_tok,
                                  const int32_t* cu_seqlens, int32_t n_seq, scone_decode* state,
                                  const int32_t* seq_slot, scone_bf16* out, int32_t* row,
                                  uint8_t* len, void* stream) {
  if (!tb || n_tok < 0 || n_seq < 0 || n_tok > 0x7FFFFFFFll) return SCONE_ERR_INVALID_ARG;
  if (n_seq == 0) return n_tok == 0 ? SCONE_OK : SCONE_ERR_INVALID_ARG;
  if (!cu_seqlens || ((uintptr_t)cu_seqlens & 3)) return SCONE_ERR_INVALID_ARG;
  if (state && (state->table != tb || (seq_slot && ((uintptr_t)seq_slot & 3)) ||
                (!seq_slot && n_seq > state->S)))
    return SCONE_ERR_INVALID_ARG;
  if (n_tok > 0 && (!tok || !out || ((uintptr_t)tok & 3) || ((uintptr_t)out & 1) ||
                    (row && ((uintptr_t)row & 3))))
    return SCONE_ERR_INVALID_ARG;
  DeviceGuard g(tb->device);
  cudaStream_t s = (cudaStream_t)stream;
  const int32_t* hist = state ? state->hist : nullptr;
  const int32_t* hlen = state ? state->hist_len : nullptr;
  const int32_t* slot = state ? seq_slot : nullptr;
  const int32_t S = state ? state->S : 0;
  const int32_t H = state ? state->H : 0;
  if (n_tok > 0) {
    const int width = row_copy_width(tb->view, out);
    const VarlenFn fn = width == 16 ? pick_varlen_w<16>(tb->fmt, tb->view.K)
                                    : pick_varlen_w<0>(tb->fmt, tb->view.K);
    const int64_t want = (n_tok + kVWarps * 8 - 1) / (kVWarps * 8);
    const int64_t cap = (int64_t)sm_count() * blocks_per_sm((const void*)fn, kVThreads, 0);
    const int grid = (int)(want < cap ? (want < 1 ? 1 : want) : cap);
    fn<<<grid, kVThreads, 0, s>>>(tb->view, tok, n_tok, cu_seqlens, n_seq, hist, hlen, slot, S,
                                  H, reinterpret_cast<uint8_t*>(out), row, len, width);
    if (cudaGetLastError() != cudaSuccess) return SCONE_ERR_CUDA;
  }
  if (state && H > 0) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((n_seq + 255) / 256));
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, varlen_hist_kernel, tok, n_tok, cu_seqlens, n_seq, state->hist,
                           state->hist_len, slot, S, H) != cudaSuccess) {
      cudaGetLastError();
      return SCONE_ERR_CUDA;
    }
  }
  return SCONE_OK;
}
