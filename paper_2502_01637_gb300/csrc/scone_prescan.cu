// Training-time pre-scan of a corpus in host memory (Appendix F: every
// training token tagged with the length and row of its longest f-gram),
// staged through HBM.
//
// scone_match can read tokens and write tags in host memory directly
// (zero-copy), but then every position's chain of dependent reads starts
// with a host-link read and the link carries scattered 4- and 1-byte
// accesses. Here the corpus moves in chunks of whole sequences: a copy engine
// brings chunk i into HBM while the match kernel tags chunk i-1 in HBM (with
// the walk over the suffix index where the table has one) and another copy
// engine returns the tags of chunk i-2, so the link runs plain bulk copies in
// both directions at once and the kernel sees device memory. Two sets of
// device buffers alternate; events order each buffer's reuse after the work
// that last read it.
//
// The buffers, streams and events are made by the first call on a table and
// kept with it (grown when a call needs larger chunks), so later calls
// allocate nothing: allocating and freeing a gigabyte per call made the call
// time vary from 33 to more than 100 ms.

#include <cstdint>
#include <new>

#include "scone_host.h"

namespace scone {

struct PrescanWork {
  int64_t chunk = 0;                 // tokens each buffer set holds
  bool with_len = false;
  int32_t* tok[2] = {nullptr, nullptr};
  int32_t* row[2] = {nullptr, nullptr};
  uint8_t* len[2] = {nullptr, nullptr};
  cudaEvent_t in_done[2] = {nullptr, nullptr};     // tokens of the chunk copied in
  cudaEvent_t match_done[2] = {nullptr, nullptr};  // kernel done (tokens free, tags ready)
  cudaEvent_t out_done[2] = {nullptr, nullptr};    // tags copied out (tag buffers free)
  cudaEvent_t start = nullptr, done = nullptr;
  cudaStream_t s_in = nullptr, s_k = nullptr, s_out = nullptr;
};

namespace {

void free_buffers(PrescanWork* w) {
  for (int i = 0; i < 2; ++i) {
    if (w->tok[i]) cudaFree(w->tok[i]);
    if (w->row[i]) cudaFree(w->row[i]);
    if (w->len[i]) cudaFree(w->len[i]);
    w->tok[i] = w->row[i] = nullptr;
    w->len[i] = nullptr;
  }
  w->chunk = 0;
  w->with_len = false;
}

// The table's workspace with buffers for `chunk` tokens (and len buffers if
// asked for); created or grown as needed. Returns SCONE_OK, NOMEM or CUDA.
int workspace(scone_table* tb, int64_t chunk, bool with_len, PrescanWork** out) {
  PrescanWork* w = tb->prescan;
  if (!w) {
    w = new (std::nothrow) PrescanWork();
    if (!w) return SCONE_ERR_NOMEM;
    bool ok = cudaStreamCreateWithFlags(&w->s_in, cudaStreamNonBlocking) == cudaSuccess &&
              cudaStreamCreateWithFlags(&w->s_k, cudaStreamNonBlocking) == cudaSuccess &&
              cudaStreamCreateWithFlags(&w->s_out, cudaStreamNonBlocking) == cudaSuccess &&
              cudaEventCreateWithFlags(&w->start, cudaEventDisableTiming) == cudaSuccess &&
              cudaEventCreateWithFlags(&w->done, cudaEventDisableTiming) == cudaSuccess;
    for (int i = 0; ok && i < 2; ++i)
      ok = cudaEventCreateWithFlags(&w->in_done[i], cudaEventDisableTiming) == cudaSuccess &&
           cudaEventCreateWithFlags(&w->match_done[i], cudaEventDisableTiming) == cudaSuccess &&
           cudaEventCreateWithFlags(&w->out_done[i], cudaEventDisableTiming) == cudaSuccess;
    if (!ok) {
      cudaGetLastError();
      prescan_release(w);
      return SCONE_ERR_CUDA;
    }
    tb->prescan = w;
  }
  if (w->chunk < chunk || (with_len && !w->with_len)) {
    free_buffers(w);
    for (int i = 0; i < 2; ++i) {
      if (cudaMalloc(&w->tok[i], (size_t)chunk * 4) != cudaSuccess ||
          cudaMalloc(&w->row[i], (size_t)chunk * 4) != cudaSuccess ||
          (with_len && cudaMalloc(&w->len[i], (size_t)chunk) != cudaSuccess)) {
        cudaGetLastError();
        free_buffers(w);
        return SCONE_ERR_NOMEM;
      }
    }
    w->chunk = chunk;
    w->with_len = with_len;
  }
  *out = w;
  return SCONE_OK;
}

}  // namespace

void prescan_release(PrescanWork* w) {
  if (!w) return;
  for (cudaStream_t s : {w->s_in, w->s_k, w->s_out})
    if (s) cudaStreamSynchronize(s);
  free_buffers(w);
  for (int i = 0; i < 2; ++i)
    for (cudaEvent_t e : {w->in_done[i], w->match_done[i], w->out_done[i]})
      if (e) cudaEventDestroy(e);
  for (cudaEvent_t e : {w->start, w->done})
    if (e) cudaEventDestroy(e);
  for (cudaStream_t s : {w->s_in, w->s_k, w->s_out})
    if (s) cudaStreamDestroy(s);
  delete w;
}

}  // namespace scone

using namespace scone;

extern "C" int scone_prescan(scone_table* tb, const int32_t* tok, int64_t B, int32_t L,
                             int32_t* row, uint8_t* len, int64_t chunk_tokens, void* stream) {
  if (!tb || B < 0 || L < 1 || chunk_tokens < 0) return SCONE_ERR_INVALID_ARG;
  const int64_t n = B * (int64_t)L;
  if (n == 0) return SCONE_OK;
  if (!tok || !row || ((uintptr_t)tok & 3) || ((uintptr_t)row & 3)) return SCONE_ERR_INVALID_ARG;
  if (chunk_tokens == 0) chunk_tokens = 32ll << 20;
  // whole sequences per chunk, at least one, and one chunk's B * L within int32
  int64_t seqs = chunk_tokens / L;
  if (seqs < 1) seqs = 1;
  if (seqs > B) seqs = B;
  if (seqs * (int64_t)L > 0x7FFFFFFFll) seqs = 0x7FFFFFFFll / L;
  if (seqs < 1) return SCONE_ERR_INVALID_ARG;
  const int64_t chunk = seqs * (int64_t)L;
  DeviceGuard g(tb->device);
  cudaStream_t caller = (cudaStream_t)stream;
  PrescanWork* w = nullptr;
  int rc = workspace(tb, chunk, len != nullptr, &w);
  if (rc != SCONE_OK) return rc;
  do {
    // work already queued on the caller's stream (the corpus being filled in,
    // for instance) comes first; so does every stage of the previous call
    if (cudaEventRecord(w->start, caller) != cudaSuccess ||
        cudaStreamWaitEvent(w->s_in, w->start, 0) != cudaSuccess) {
      rc = SCONE_ERR_CUDA;
      break;
    }
    int k = 0;
    for (int64_t off = 0; off < n; off += chunk, ++k) {
      const int b = k & 1;
      const int64_t m = n - off < chunk ? n - off : chunk;
      // tokens in, once the kernel two chunks back has read this buffer
      if ((k >= 2 && cudaStreamWaitEvent(w->s_in, w->match_done[b], 0) != cudaSuccess) ||
          cudaMemcpyAsync(w->tok[b], tok + off, (size_t)m * 4, cudaMemcpyHostToDevice,
                          w->s_in) != cudaSuccess ||
          cudaEventRecord(w->in_done[b], w->s_in) != cudaSuccess) {
        rc = SCONE_ERR_CUDA;
        break;
      }
      // the match, once the tokens are in and the tags two chunks back are out
      if (cudaStreamWaitEvent(w->s_k, w->in_done[b], 0) != cudaSuccess ||
          (k >= 2 && cudaStreamWaitEvent(w->s_k, w->out_done[b], 0) != cudaSuccess)) {
        rc = SCONE_ERR_CUDA;
        break;
      }
      rc = scone_match(tb, w->tok[b], (int32_t)(m / L), L, w->row[b], len ? w->len[b] : nullptr,
                       w->s_k);
      if (rc != SCONE_OK) break;
      if (cudaEventRecord(w->match_done[b], w->s_k) != cudaSuccess ||
          cudaStreamWaitEvent(w->s_out, w->match_done[b], 0) != cudaSuccess ||
          cudaMemcpyAsync(row + off, w->row[b], (size_t)m * 4, cudaMemcpyDeviceToHost,
                          w->s_out) != cudaSuccess ||
          (len && cudaMemcpyAsync(len + off, w->len[b], (size_t)m, cudaMemcpyDeviceToHost,
                                  w->s_out) != cudaSuccess) ||
          cudaEventRecord(w->out_done[b], w->s_out) != cudaSuccess) {
        rc = SCONE_ERR_CUDA;
        break;
      }
    }
    if (rc != SCONE_OK) break;
    // the caller's stream continues after the last tags are out; the next
    // call's first copies wait on the caller's stream, so they also follow
    // this call's last kernel and copies
    if (cudaEventRecord(w->done, w->s_out) != cudaSuccess ||
        cudaStreamWaitEvent(caller, w->done, 0) != cudaSuccess)
      rc = SCONE_ERR_CUDA;
  } while (0);
  if (rc != SCONE_OK) {
    cudaGetLastError();
    // leave nothing queued on the buffers
    cudaStreamSynchronize(w->s_in);
    cudaStreamSynchronize(w->s_k);
    cudaStreamSynchronize(w->s_out);
    return rc;
  }
  // the tags are in host memory when the call returns
  return cudaStreamSynchronize(caller) == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}
