// The tensor-core GEMM of the f-gram model (scone_gemm.cu), for the other
// translation units of the library.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "scone.h"

namespace scone {

enum GemmEpilogue {
  GEMM_EPI_STORE = SCONE_GEMM_STORE,        // C = A B^T
  GEMM_EPI_RESIDUAL = SCONE_GEMM_RESIDUAL,  // C = R + A B^T (C may be R)
  GEMM_EPI_SWIGLU = SCONE_GEMM_SWIGLU       // C[:, j] = silu(gate_j) up_j, C is [M x N/2]
};

// C[M x N] = epilogue(A[M x K] . B[N x K]^T), bf16 row-major, K contiguous;
// N a multiple of 256, K of 64, pointers 16-byte aligned. Device-detected
// failures (a pipeline wait that timed out) set *status to SCONE_ERR_CUDA.
int gemm_bf16(const uint16_t* A, const uint16_t* B, const uint16_t* R, uint16_t* C, int M, int N,
              int K, int epi, int* status, cudaStream_t s);

// The same with the kernel chosen: 0 = default (SM pairs), 1 = one SM per
// 128 x 256 tile, 2 = SM pairs (256 x 256 tiles, tcgen05 cta_group::2).
int gemm_bf16_variant(const uint16_t* A, const uint16_t* B, const uint16_t* R, uint16_t* C,
                      int M, int N, int K, int epi, int variant, int* status, cudaStream_t s);

}  // namespace scone
