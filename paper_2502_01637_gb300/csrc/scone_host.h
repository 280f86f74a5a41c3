// Host-side state shared by the C ABI translation units.
#pragma once

#include <cstdint>
#include <vector>
#include <cuda_runtime.h>

#include "scone.h"
#include "scone_device.cuh"

namespace scone {
struct PrescanWork;   // scone_prescan's device buffers, streams and events (scone_prescan.cu)
void prescan_release(PrescanWork* w);
}  // namespace scone

struct scone_table {
  int device = 0;
  int fmt = scone::FMT16;
  uint8_t* slots = nullptr;  // n_buckets * 32 bytes
  int* status = nullptr;     // sticky device error word
  int* status_host = nullptr;      // pinned, device-mapped [2]: the recorded error's copy and
                                   // the fetched status word, read by scone_status
  int* status_host_dev = nullptr;  // its device address
  uint8_t* zero_row = nullptr;  // d * 2 zero bytes: the source of error positions (bulk copies)
  int copy_mode = SCONE_COPY_AUTO;
  scone::PrescanWork* prescan = nullptr;  // made by the first scone_prescan call, kept
  scone::TableView view{};
  scone_table_info info{};
};

struct scone_decode {
  const scone_table* table = nullptr;
  int32_t S = 0;
  int32_t H = 0;             // history length kept per sequence (K - 1)
  int32_t* hist = nullptr;   // device [S * H], right-aligned, oldest first
  int32_t* hist_len = nullptr;  // device [S]
};

namespace scone {

// Device-current guard: switches to the table's device for the call.
struct DeviceGuard {
  int prev = -1;
  int want = -1;
  explicit DeviceGuard(int dev) : want(dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
  }
  ~DeviceGuard() {
    if (prev >= 0 && prev != want) cudaSetDevice(prev);
  }
};

// Suffix index of an f-gram list (scone_suffix.cu): ext[r] = 1 when f-gram
// r is the suffix of a longer listed f-gram; the markers are the suffixes
// (length >= 2) of listed f-grams that are not listed themselves, each once
// ([n_markers x K] tokens padded with -1, and their lengths). Returns
// SCONE_OK, DUPLICATE_FGRAM, UNSUPPORTED (too many entries) or NOMEM.
struct SuffixIndex {
  std::vector<uint8_t> ext;
  std::vector<int32_t> marker_tok;
  std::vector<uint8_t> marker_len;
  int64_t n_markers = 0;
};
int suffix_index(const int32_t* tok, const uint8_t* len, int64_t n, int K, SuffixIndex* out);

// Whether a table of this key format and K gets a suffix index at build:
// the kernels that walk the lengths (the pipelined embed) take 16-byte slots
// and K <= 5; for K = 2 there are no suffixes to index.
inline bool wants_suffix_index(int fmt, int K) { return fmt == FMT16 && K >= 3 && K <= 5; }

// Bulk (TMA) fused embed: eligibility for a call and launch.
bool bulk_eligible(const scone_table* tb, const void* out);
int launch_embed_bulk(const scone_table* tb, const int32_t* tok, int64_t n, int32_t L,
                      uint8_t* out, int32_t* row, uint8_t* len, cudaStream_t stream);

// Fused embed with separate match and copy warps (SCONE_COPY_SPLIT): launch.
int launch_embed_split(const scone_table* tb, const int32_t* tok, int64_t n, int32_t L,
                       uint8_t* out, int32_t* row, uint8_t* len, cudaStream_t stream);

// Fused embed with the next tile's match interleaved into the copy
// (SCONE_COPY_PIPELINED): eligibility (FMT16, K <= 5, 16-byte copies) and launch.
bool pipe_eligible(const scone_table* tb, const void* out);
int launch_embed_pipe(const scone_table* tb, const int32_t* tok, int64_t n, int32_t L,
                      uint8_t* out, int32_t* row, uint8_t* len, cudaStream_t stream);

// Widest copy unit (16, 8, 4 or 2 bytes) that the row size, T, F, the output
// and `extra` (another base address or size, 0 if none) all allow.
inline int row_copy_width(const TableView& t, const void* out, uintptr_t extra = 0) {
  uintptr_t a = (uintptr_t)t.T | (uintptr_t)out | (uintptr_t)(t.d * 2) | extra;
  if (t.n_fgrams > 0) a |= (uintptr_t)t.F;
  if ((a & 15) == 0) return 16;
  if ((a & 7) == 0) return 8;
  if ((a & 3) == 0) return 4;
  return 2;
}

// Resident blocks per SM for a kernel at a block size (cached per function).
int blocks_per_sm(const void* fn, int threads, size_t smem);
int sm_count();

}  // namespace scone
