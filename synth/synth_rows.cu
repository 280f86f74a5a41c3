// Device-side fill of seeded bf16 embedding rows (input generation only).
//
// Computes, for every element, the same Irwin-Hall(4) draw as the host
// function synth_rows_cpu in synth.cpp: SplitMix64 counter draw, sum of the
// four 16-bit quarters, one fp32 multiply, bf16 round-to-nearest-even. All
// steps are integer or a single IEEE multiply, so the bytes match the host's.
// The destination may be device memory or host-pinned, device-mapped memory.

#include <cstdint>
#include <cuda_runtime.h>

namespace {

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint16_t row_element(uint64_t seed, uint64_t ctr) {
  const uint64_t x = mix64(seed + (ctr + 1) * 0x9E3779B97F4A7C15ull);
  const int32_t s = (int32_t)(x & 0xFFFF) + (int32_t)((x >> 16) & 0xFFFF) +
                    (int32_t)((x >> 32) & 0xFFFF) + (int32_t)(x >> 48) - 131070;
  const float v = __fmul_rn((float)s, 0x1.1bc77ap-21f);
  uint32_t u = __float_as_uint(v);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

// One thread writes 8 consecutive elements of the flattened [n x d] block.
__global__ void rows_fill_kernel(uint64_t seed, int32_t d, int64_t row0, int64_t n_elem,
                                 uint16_t* __restrict__ out) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x * 8;
  for (int64_t e = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 8; e < n_elem; e += stride) {
    const uint64_t base = (uint64_t)row0 * (uint64_t)d + (uint64_t)e;
    if (e + 8 <= n_elem) {
      uint32_t w[4];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        w[j] = (uint32_t)row_element(seed, base + 2 * j) |
               ((uint32_t)row_element(seed, base + 2 * j + 1) << 16);
      *reinterpret_cast<uint4*>(out + e) = make_uint4(w[0], w[1], w[2], w[3]);
    } else {
      for (int64_t k = e; k < n_elem; ++k) out[k] = row_element(seed, base + (k - e));
    }
  }
}

}  // namespace

extern "C" int synth_rows_gpu(uint64_t seed, int32_t d, int64_t row0, int64_t n, uint16_t* out,
                              void* stream) {
  if (d <= 0 || n < 0 || row0 < 0) return -1;
  if (n == 0) return 0;
  if ((reinterpret_cast<uintptr_t>(out) & 15) != 0) return -1;
  const int64_t n_elem = n * (int64_t)d;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  int64_t blocks = (n_elem / 8 + 255) / 256;
  const int64_t cap = (int64_t)(sms > 0 ? sms : 1) * 16;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  rows_fill_kernel<<<(unsigned)blocks, 256, 0, (cudaStream_t)stream>>>(seed, d, row0, n_elem, out);
  return cudaGetLastError() == cudaSuccess ? 0 : -7;
}
