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
// (the last b with cu[b] <= p, so empty sequences are skipped), and window
// tokens left of the chunk come from the history. A warp finds the sequence
// of its first position with a 32-way search by all its lanes; later
// positions gallop from the sequence of the warp's previous tile.
//
// The history update (each continued slot's history becomes the last K-1
// tokens of history ++ chunk) happens in the same launch, without waiting on
// other blocks. Only a chunk's first min(c, K-1) positions read the slot's
// old history (its readers). The warp ranges are shifted so that no chunk's
// readers straddle two warps, and the lane of a chunk's last reader writes
// the new history after a __syncwarp that orders it behind the other
// readers' loads; readers in earlier tiles of the warp came before it.
//
// On a table with a suffix index (16-byte slots, K <= 5, 16-byte copies)
// varlen_walk_kernel takes the place of varlen_embed_kernel: the walk over
// the lengths of scone_walk.cuh, interleaved into the row copy as in
// embed_walk_kernel, with each lane's window built as above.

#include "scone_host.h"
#include "scone_walk.cuh"

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

// The same answer (last b with cu[b] <= q, q >= 0) found by a whole warp:
// each round the 32 lanes read evenly spaced entries of the range still open
// and a ballot keeps the piece that holds the answer (cu is nondecreasing, so
// the lanes that pass form a prefix). n_seq sequences take ceil(log32 n_seq)
// dependent reads instead of about 2 log2 n_seq. Warp-uniform call.
__device__ __forceinline__ int32_t warp_seq(const int32_t* __restrict__ cu, int32_t n_seq,
                                            int64_t q, int lane) {
  int32_t lo = 0, hi = n_seq - 1;
  while (lo < hi) {
    const int32_t step = (hi - lo + 31) / 32;
    const int32_t probe = lo + 1 + lane * step;
    const bool ok = probe <= hi && (int64_t)__ldg(cu + probe) <= q;
    const int k = __popc(__ballot_sync(0xFFFFFFFFu, ok));
    if (k == 0) {
      hi = lo;
    } else {
      lo += 1 + (k - 1) * step;
      const int32_t top = lo + step - 1;
      hi = top < hi ? top : hi;
    }
  }
  return lo;
}

// A warp-range boundary q moved past the readers of the chunk it would cut:
// if q falls inside the first min(c, H) positions of a chunk (other than at
// its start), the boundary moves to their end. Monotone in q, so the moved
// ranges still tile [0, n_tok). Warp-uniform call.
__device__ __forceinline__ int64_t reader_bound(int64_t q, int64_t n_tok,
                                                const int32_t* __restrict__ cu, int32_t n_seq,
                                                int32_t H, int lane) {
  if (q <= 0 || q >= n_tok) return q;
  const int32_t b = warp_seq(cu, n_seq, q, lane);
  const int64_t c0 = __ldg(cu + b), c = (int64_t)__ldg(cu + b + 1) - c0;
  const int64_t m = c < H ? c : H;
  return (c0 < q && q < c0 + m) ? c0 + m : q;
}

// Positions [lo, hi) of warp w of nw: an even split, with the boundaries
// moved by reader_bound when the launch continues a decode state.
__device__ __forceinline__ void varlen_warp_range(int64_t n_tok, int64_t w, int64_t nw,
                                                  const int32_t* __restrict__ cu, int32_t n_seq,
                                                  bool readers, int32_t H, int lane,
                                                  int64_t* lo, int64_t* hi) {
  *lo = n_tok * w / nw;
  *hi = n_tok * (w + 1) / nw;
  if (readers) {
    *lo = reader_bound(*lo, n_tok, cu, n_seq, H, lane);
    *hi = reader_bound(*hi, n_tok, cu, n_seq, H, lane);
  }
}

// Where packed position p of sequence b sits: the chunk's start c0 and
// length c, the offset i in the chunk, and with a decode state the slot s
// (-1 if outside [0, S)) and the history length h its window may use
// (only the chunk's first K-1 positions reach into the history).
struct VarPos {
  int32_t b, s, h, c0, c, i;
  const int32_t* hrow;
};

__device__ __forceinline__ VarPos locate(const TableView& t, const int32_t* __restrict__ cu,
                                         const int32_t* hist, const int32_t* hist_len,
                                         const int32_t* __restrict__ slot, int32_t S, int32_t H,
                                         int64_t p, int32_t b) {
  VarPos v;
  v.b = b;
  v.c0 = __ldg(cu + v.b);
  v.c = __ldg(cu + v.b + 1) - v.c0;
  v.i = (int32_t)(p - (v.c0 > 0 ? v.c0 : 0));   // offset in the chunk, never left of tok[0]
  v.s = -1;
  v.h = 0;
  v.hrow = nullptr;
  if (hist) {
    const int32_t s = slot ? __ldg(slot + v.b) : v.b;
    if (s >= 0 && s < S) {
      v.s = s;
      if (v.i < t.K - 1) v.h = hist_len[s];
      v.hrow = hist + (int64_t)s * H;
    }
  }
  return v;
}

// The slot this lane rewrites the history of, or -1: the lane of a chunk's
// last reader (offset min(c, H) - 1) of a valid slot and a well-formed chunk.
__device__ __forceinline__ int32_t history_writer(const VarPos& v, int64_t n_tok, int32_t H) {
  if (v.s < 0 || v.c0 < 0 || (int64_t)v.c0 + v.c > n_tok) return -1;
  const int32_t m = v.c < H ? v.c : H;
  return v.i == m - 1 ? v.s : -1;
}

// Slot s's history becomes the last H tokens of history ++ chunk
// (right-aligned, oldest first; the chunk is tok[c0 .. c0 + c)), its
// length min(H, h + c).
__device__ __forceinline__ void write_history(const int32_t* __restrict__ tok, int32_t s,
                                              int32_t c0, int32_t c, int32_t* hist,
                                              int32_t* hist_len, int32_t H) {
  int32_t* row = hist + (int64_t)s * H;
  const int32_t h = hist_len[s];
  int32_t nw[7];                           // H <= 7
#pragma unroll
  for (int j = 0; j < 7; ++j) {
    if (j < H) {
      // entry j of the new row is the token H - j places from the end of
      // history ++ chunk
      const int32_t back = H - j;          // 1 = the chunk's last token
      nw[j] = back <= c ? __ldg(tok + c0 + c - back) : row[H - (back - c)];
    }
  }
#pragma unroll
  for (int j = 0; j < 7; ++j)
    if (j < H) row[j] = nw[j];
  hist_len[s] = h + c < H ? h + c : H;
}

// Selection for packed position p located at v, with token x. Sets *len /
// *err like match_position; a slot outside [0, S) is SCONE_ERR_INVALID_ARG
// (reported after a bad token).
template <int FMT, int KT>
__device__ __forceinline__ int32_t match_varlen(const TableView& t,
                                                const int32_t* __restrict__ tok,
                                                const VarPos& v, bool with_state, int32_t H,
                                                int64_t p, int32_t x, int* len, int* err) {
  if (!valid_token(x, t.vocab)) {
    *err = SCONE_ERR_TOKEN_RANGE;
    *len = 0;
    return -1;
  }
  if (with_state && v.s < 0) {
    *err = SCONE_ERR_INVALID_ARG;
    *len = 0;
    return -1;
  }
  const int64_t known = (int64_t)v.i + 1 + v.h;   // tokens of the sequence up to p
  const int nmax = known < t.K ? (int)known : t.K;
  const int32_t i = v.i;
  const int32_t* hrow = v.hrow;
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
                        const int32_t* __restrict__ cu, int32_t n_seq, int32_t* hist,
                        int32_t* hist_len, const int32_t* __restrict__ slot, int32_t S, int32_t H,
                        uint8_t* __restrict__ out, int32_t* __restrict__ row_out,
                        uint8_t* __restrict__ len_out, int width) {
  __shared__ const void* src_s[kVWarps][32];
  __shared__ int3 wr_s[kVWarps][32];   // history this lane writes: slot (or -1), chunk start, length
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int row_bytes = t.d * 2;
  const bool with_state = hist != nullptr;
  int64_t lo, hi;
  varlen_warp_range(n_tok, (int64_t)blockIdx.x * kVWarps + warp, (int64_t)gridDim.x * kVWarps,
                    cu, n_seq, with_state, H, lane, &lo, &hi);
  if (lo >= hi) return;
  int32_t bq = warp_seq(cu, n_seq, lo, lane);   // sequence of the warp's previous position
  for (int64_t base = lo; base < hi; base += 32) {
    const int nrows = (int)(hi - base < 32 ? hi - base : 32);
    const int64_t p = base + lane;
    const void* src = nullptr;
    VarPos v;
    const int32_t b = lane < nrows ? seq_from(cu, n_seq, p, bq) : bq;
    if (lane < nrows) v = locate(t, cu, hist, hist_len, slot, S, H, p, b);
    bq = __shfl_sync(0xFFFFFFFFu, b, nrows - 1);
    if (lane < nrows) {
      const int32_t x = __ldg(tok + p);
      int len = 0, err = 0;
      const int32_t r = match_varlen<FMT, KT>(t, tok, v, with_state, H, p, x, &len, &err);
      if (err) {
        record_error(t, err);
      } else {
        src = r >= 0 ? static_cast<const void*>(t.F + (int64_t)r * t.d)
                     : static_cast<const void*>(t.T + (int64_t)x * t.d);
      }
      if (row_out) row_out[p] = r;
      if (len_out) len_out[p] = (uint8_t)len;
      if (with_state) wr_s[warp][lane] = make_int3(history_writer(v, n_tok, H), v.c0, v.c);
    } else if (with_state) {
      wr_s[warp][lane].x = -1;
    }
    src_s[warp][lane] = src;
    __syncwarp();   // also orders the readers' history loads before the writer's stores
    if (with_state) {
      const int3 wr = wr_s[warp][lane];
      if (wr.x >= 0) write_history(tok, wr.x, wr.y, wr.z, hist, hist_len, H);
    }
    warp_copy_rows_w<W, VarlenTuning<KT>::kLoads>(src_s[warp], out + base * (int64_t)row_bytes,
                                                  nrows, row_bytes, width, lane);
    __syncwarp();
  }
}

// The positions [lo, hi) of one warp of varlen_walk_kernel: the walk schedule
// of embed_walk_kernel (scone_pipe.cu) over packed sequences. A warp's first
// tile of kWalkFirst positions is walked before its copy, then each next
// tile's rounds run between the chunks of the current tile's copy; lane
// state, errors and history writes as in varlen_embed_kernel.
template <int KT>
__device__ __forceinline__ void varlen_walk_positions(
    const TableView& t, const int32_t* __restrict__ tok, int64_t n_tok,
    const int32_t* __restrict__ cu, int32_t n_seq, int32_t* hist, int32_t* hist_len,
    const int32_t* __restrict__ slot, int32_t S, int32_t H, uint8_t* __restrict__ out,
    int32_t* __restrict__ row_out, uint8_t* __restrict__ len_out, int64_t lo, int64_t hi,
    int lane, int warp) {
  constexpr int U = kWalkLoads;
  __shared__ const uint4* src_s[kVWarps][2][32];
  __shared__ __align__(16) Bucket bucket_s[kVWarps][32];
  __shared__ int3 wr_s[kVWarps][32];   // history this lane writes: slot (or -1), chunk start, length
  const int epr = t.d >> 3;                      // 16-byte elements per row
  const bool with_state = hist != nullptr;
  PipeWalk<KT> m;
  m.sb = &bucket_s[warp][lane];
  int32_t bq = warp_seq(cu, n_seq, lo, lane);   // sequence of the warp's previous position
  // starts the walks of positions [tb, tb + nn), one per lane (warp-uniform call)
  auto begin = [&](int64_t tb, int nn) {
    const int64_t p = tb + lane;
    const bool act = lane < nn;
    VarPos v;
    const int32_t b = act ? seq_from(cu, n_seq, p, bq) : bq;
    if (act) v = locate(t, cu, hist, hist_len, slot, S, H, p, b);
    bq = __shfl_sync(0xFFFFFFFFu, b, nn - 1);
    if (!act) {
      if (with_state) wr_s[warp][lane].x = -1;
      m.start_with(false, 0, 0, 0, [](int) { return 0; });
      return;
    }
    if (with_state) wr_s[warp][lane] = make_int3(history_writer(v, n_tok, H), v.c0, v.c);
    const int64_t known = (int64_t)v.i + 1 + v.h;   // tokens of the sequence up to p
    const int nm = known < t.K ? (int)known : t.K;
    const int32_t i = v.i;
    const int32_t* hrow = v.hrow;
    m.start_with(true, __ldg(tok + p), nm, with_state && v.s < 0 ? SCONE_ERR_INVALID_ARG : 0,
                 [&](int j) { return j <= i ? __ldg(tok + p - j) : hrow[H - (j - i)]; });
  };
  // after a tile's rounds: its readers have loaded their windows
  auto history = [&]() {
    __syncwarp();
    if (with_state) {
      const int3 wr = wr_s[warp][lane];
      if (wr.x >= 0) write_history(tok, wr.x, wr.y, wr.z, hist, hist_len, H);
    }
  };
  int buf = 0;
  int64_t base = lo;
  int nrows = (int)(hi - base < kWalkFirst ? hi - base : kWalkFirst);
  begin(base, nrows);
  while (__any_sync(0xFFFFFFFFu, m.state != 0)) m.round(t);
  src_s[warp][buf][lane] =
      lane < nrows ? walk_finish<KT>(t, m, base + lane, row_out, len_out) : nullptr;
  history();
  __syncwarp();
  while (base < hi) {
    const int64_t nbase = base + nrows;
    const int nn = nbase < hi ? (int)(hi - nbase < 32 ? hi - nbase : 32) : 0;
    const int64_t total = (int64_t)nrows * epr;
    const int nchunks = (int)((total + 32 * U - 1) / (32 * U));
    const uint4* const* src = src_s[warp][buf];
    uint4* dst = reinterpret_cast<uint4*>(out) + base * epr;
    int r = 0, col = lane;
    while (col >= epr) {
      col -= epr;
      ++r;
    }
    if (nn) begin(nbase, nn);
    for (int c = 0; c < nchunks; ++c) {
      copy_chunks<U>(src, dst, nrows, epr, total, lane, c, c + 1, r, col);
      if (nn) m.round(t);
    }
    if (nn) {
      while (__any_sync(0xFFFFFFFFu, m.state != 0)) m.round(t);
      src_s[warp][buf ^ 1][lane] =
          lane < nn ? walk_finish<KT>(t, m, nbase + lane, row_out, len_out) : nullptr;
      history();
    }
    __syncwarp();
    buf ^= 1;
    base = nbase;
    nrows = nn;
  }
}

template <int KT>
__global__ void __launch_bounds__(kVThreads, kWalkMinBlocks)
    varlen_walk_kernel(const TableView t, const int32_t* __restrict__ tok, int64_t n_tok,
                       const int32_t* __restrict__ cu, int32_t n_seq, int32_t* hist,
                       int32_t* hist_len, const int32_t* __restrict__ slot, int32_t S, int32_t H,
                       uint8_t* __restrict__ out, int32_t* __restrict__ row_out,
                       uint8_t* __restrict__ len_out) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int64_t lo, hi;
  varlen_warp_range(n_tok, (int64_t)blockIdx.x * kVWarps + warp, (int64_t)gridDim.x * kVWarps,
                    cu, n_seq, hist != nullptr, H, lane, &lo, &hi);
  if (lo < hi)
    varlen_walk_positions<KT>(t, tok, n_tok, cu, n_seq, hist, hist_len, slot, S, H, out, row_out,
                              len_out, lo, hi, lane, warp);
}

using VarlenFn = void (*)(TableView, const int32_t*, int64_t, const int32_t*, int32_t, int32_t*,
                          int32_t*, const int32_t*, int32_t, int32_t, uint8_t*, int32_t*,
                          uint8_t*, int);
using VarlenWalkFn = void (*)(TableView, const int32_t*, int64_t, const int32_t*, int32_t,
                              int32_t*, int32_t*, const int32_t*, int32_t, int32_t, uint8_t*,
                              int32_t*, uint8_t*);

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

// The walk applies: suffix index, the default probe limit, 16-byte slots,
// K <= 5, 16-byte copies, and a copy mode of AUTO or PIPELINED (REGISTERS
// keeps varlen_embed_kernel; BULK and SPLIT have no ragged variant).
bool varlen_walk_eligible(const scone_table* tb, const void* out) {
  return tb->view.suffix_index && tb->view.probe_limit >= 2 && pipe_eligible(tb, out) &&
         (tb->copy_mode == SCONE_COPY_AUTO || tb->copy_mode == SCONE_COPY_PIPELINED);
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
  if (n_tok == 0) return SCONE_OK;   // every chunk is empty: no row and no history changes
  DeviceGuard g(tb->device);
  cudaStream_t s = (cudaStream_t)stream;
  // with a state the kernels read the slots' histories and rewrite them in place
  int32_t* hist = state && state->H > 0 ? state->hist : nullptr;
  int32_t* hlen = state && state->H > 0 ? state->hist_len : nullptr;
  const int32_t* slot = hist ? seq_slot : nullptr;
  const int32_t S = hist ? state->S : 0;
  const int32_t H = hist ? state->H : 0;
  const int64_t want = (n_tok + kVWarps * 8 - 1) / (kVWarps * 8);
  if (varlen_walk_eligible(tb, out)) {
    const VarlenWalkFn fn = tb->view.K <= 3 ? varlen_walk_kernel<3> : varlen_walk_kernel<5>;
    const int64_t cap = (int64_t)sm_count() * blocks_per_sm((const void*)fn, kVThreads, 0);
    const int grid = (int)(want < cap ? (want < 1 ? 1 : want) : cap);
    fn<<<grid, kVThreads, 0, s>>>(tb->view, tok, n_tok, cu_seqlens, n_seq, hist, hlen, slot, S,
                                  H, reinterpret_cast<uint8_t*>(out), row, len);
  } else {
    const int width = row_copy_width(tb->view, out);
    const VarlenFn fn = width == 16 ? pick_varlen_w<16>(tb->fmt, tb->view.K)
                                    : pick_varlen_w<0>(tb->fmt, tb->view.K);
    const int64_t cap = (int64_t)sm_count() * blocks_per_sm((const void*)fn, kVThreads, 0);
    const int grid = (int)(want < cap ? (want < 1 ? 1 : want) : cap);
    fn<<<grid, kVThreads, 0, s>>>(tb->view, tok, n_tok, cu_seqlens, n_seq, hist, hlen, slot, S,
                                  H, reinterpret_cast<uint8_t*>(out), row, len, width);
  }
  return cudaGetLastError() == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}
