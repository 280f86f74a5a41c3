// Host-side state shared by the C ABI translation units.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "scone.h"
#include "scone_device.cuh"

struct scone_table {
  int device = 0;
  int fmt = scone::FMT16;
  uint8_t* slots = nullptr;  // n_buckets * 32 bytes
  int* status = nullptr;     // sticky device error word
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

// Resident blocks per SM for a kernel at a block size (cached per function).
int blocks_per_sm(const void* fn, int threads, size_t smem);
int sm_count();

}  // namespace scone
