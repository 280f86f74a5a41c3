// bf16 GEMM on the 5th-generation tensor cores (tcgen05) for the f-gram
// model's dense layers: C[M x N] = epilogue(A[M x K] . B[N x K]^T), A and B
// row-major with K contiguous (activations x weights), fp32 accumulation in
// tensor memory.
//
// Tiles of 128 x 256, persistent (one CTA per SM walks its share of the
// tiles in a grouped order: 8192 rows of row tiles at a time sweep every column
// tile, so the tiles in flight share their A and B slices in L2),
// warp-specialized:
//   * warp 0 streams K-slices of 64 (A: 128 x 64, B: 256 x 64, 48 KB) into a
//     ring of kStages shared-memory stages with TMA (cp.async.bulk.tensor,
//     128-byte swizzle), each stage completed on an mbarrier by byte count;
//   * warp 1 issues tcgen05.mma (M = 128, N = 256, K = 16, bf16 x bf16 ->
//     fp32), four per slice, into one of two 256-column accumulators in
//     tensor memory, frees each stage with tcgen05.commit and hands a
//     finished accumulator to the epilogue with another commit;
//   * warps 2..5 read the other accumulator back with tcgen05.ld (warp w owns
//     tensor-memory lanes 32 (w % 4) .. + 31, i.e. rows) and apply the
//     epilogue: store, add a residual, or SwiGLU of interleaved gate/up
//     column pairs; they stage the bf16 results in swizzled shared-memory
//     boxes that TMA stores to C, and release the accumulator.
// So the epilogue of one tile overlaps the main loop of the next.
// Every mbarrier wait is bounded (kGemmSpin polls); past it the CTA records
// SCONE_ERR_CUDA, stops issuing, waits for what it issued, frees its tensor
// memory and returns.

#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <cstring>
#include <mutex>

#include "scone_gemm.h"
#include "scone_host.h"
#include "scone_ptx.cuh"

namespace scone {

namespace {

constexpr int kBM = 128, kBN = 256, kBK = 64;
constexpr int kStages = 4;
constexpr int kEpiWarps = 4;
constexpr int kGemmThreads = 32 * (2 + kEpiWarps);   // loader, MMA issuer, 4 epilogue warps
// Rows per group of the tile order (kGroupRows / tile height row tiles at a
// time). On M = N = 16384, K = 2048, groups of 8, 16, 32 and 64 row tiles
// gave the SM-pair kernel (256-row tiles) 1704, 1714, 1722 and 1681-1688
// TFLOP/s, and the one-SM kernel (128-row tiles) 1607, 1668, 1697 and 1741:
// both are best near 8192 rows.
constexpr int kGroupRows = 8192;
constexpr uint32_t kStageA = kBM * kBK * 2;   // 16 KB
constexpr uint32_t kStageB = kBN * kBK * 2;   // 32 KB
constexpr uint32_t kStageBytes = kStageA + kStageB;
constexpr uint32_t kTmemCols = 2 * kBN;       // two fp32 accumulators of 256 columns x 128 lanes
constexpr uint32_t kGemmSpin = 1u << 22;   // polls; each try_wait may also suspend briefly
constexpr size_t kGemmSmem = (size_t)kStages * kStageBytes + 1024 /* align */ + 256 /* barriers */ +
                             (size_t)kEpiWarps * 2 * 32 * 128 /* epilogue boxes */;

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  return mbar_wait_bounded(bar, parity, kGemmSpin);
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

// Shared-memory matrix descriptor of a K-major tile whose rows are 128 bytes
// (64 bf16) with the 128-byte swizzle: 8-row atoms of 1024 bytes, stride
// between atoms 1024 bytes; the leading-dimension offset is unused for this
// layout. Bits: start >> 4 at 0, LBO >> 4 at 16, SBO >> 4 at 32, version 1 at
// 46, swizzle mode 2 (128 B) at 61.
__device__ __forceinline__ uint64_t desc_k128(uint32_t smem_byte_addr) {
  uint64_t d = (uint64_t)((smem_byte_addr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;
  d |= (uint64_t)(1024 >> 4) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor, kind::f16: D f32 (bits 4-5 = 1), A and B bf16 (bits
// 7-9, 10-12 = 1), both K-major (bits 15, 16 = 0), N >> 3 at 17, M >> 4 at 24.
constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kBN >> 3) << 17) |
                            ((uint32_t)(kBM >> 4) << 24);

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n"
      " setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(kIdesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
      "%11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, "
      "%28, %29, %30, %31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);   // a in the low half
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// Tile t of the grouped order: G row tiles at a time sweep all column tiles,
// so the CTAs running at once share a few A tiles and a few B tiles in L2
// instead of each streaming its own A.
template <int G>
__device__ __forceinline__ void tile_coords(int t, int num_m, int num_n, int* m_tile,
                                            int* n_tile) {
  const int per_group = G * num_n;
  const int first_m = (t / per_group) * G;
  const int gm = num_m - first_m < G ? num_m - first_m : G;
  const int local = t % per_group;
  *m_tile = first_m + local % gm;
  *n_tile = local / gm;
}

// Epilogue of one 32-column chunk of one row: v holds columns c .. c+31 of
// the accumulator row.
template <int EPI>
__device__ __forceinline__ void store_chunk(const float (&v)[32], int row, int col,
                                            const uint16_t* __restrict__ R,
                                            uint16_t* __restrict__ C, int ldc) {
  if constexpr (EPI == GEMM_EPI_SWIGLU) {
    // 16 gates then 16 ups of outputs col / 2 ..
    uint32_t o[8];
#pragma unroll
    for (int j = 0; j < 16; j += 2) {
      const float g0 = v[j], g1 = v[j + 1], u0 = v[16 + j], u1 = v[17 + j];
      o[j / 2] = pack_bf16(g0 / (1.f + expf(-g0)) * u0, g1 / (1.f + expf(-g1)) * u1);
    }
    uint4* dst = reinterpret_cast<uint4*>(C + (int64_t)row * ldc + col / 2);
    dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
    dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
  } else {
    uint32_t o[16];
    if constexpr (EPI == GEMM_EPI_RESIDUAL) {
      const uint4* src = reinterpret_cast<const uint4*>(R + (int64_t)row * ldc + col);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 r4 = src[q];
        const uint32_t rw[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int j = q * 8 + e * 2;
          o[q * 4 + e] = pack_bf16(v[j] + bf16_lo(rw[e]), v[j + 1] + bf16_hi(rw[e]));
        }
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; j += 2) o[j / 2] = pack_bf16(v[j], v[j + 1]);
    }
    uint4* dst = reinterpret_cast<uint4*>(C + (int64_t)row * ldc + col);
#pragma unroll
    for (int q = 0; q < 4; ++q)
      dst[q] = make_uint4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
  }
}

// The epilogue writes C through shared memory and TMA: each epilogue warp
// stages its 32 rows of 64 output columns (128 bytes a row: two 32-column
// chunks of the accumulator, or four under SwiGLU, whose output is half as
// wide) as a box [32 rows x 128 bytes] with the 128-byte swizzle (16-byte
// unit u of row r at unit u ^ (r % 8), so the lanes' row writes spread over
// the banks), and one lane stores the box with cp.async.bulk.tensor. C is
// then written in whole 128-byte lines instead of 32 scattered pieces per
// warp store. Two boxes per warp alternate; a box is rewritten only after
// the store that read it has finished reading (bulk wait_group.read 1).
// Rows past M are clipped by the store.
constexpr uint32_t kEpiBox = 32 * 128;                        // bytes per staged box
constexpr uint32_t kEpiSmem = kEpiWarps * 2 * kEpiBox;        // 32 KB per CTA
constexpr int kEpiBoxCols = 64;                               // bf16 output columns per box
template <int EPI>
__host__ __device__ constexpr int epi_chunks_per_box() {
  return EPI == GEMM_EPI_SWIGLU ? 4 : 2;
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap* map, uint32_t src, int x, int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(x), "r"(y), "r"(src)
      : "memory");
}
__device__ __forceinline__ void epi_commit() { asm volatile("cp.async.bulk.commit_group;"); }
__device__ __forceinline__ void epi_wait_read_1() {
  asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
__device__ __forceinline__ void epi_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// This lane's row of one chunk (accumulator columns col .. col+31) as the
// epilogue's bf16 output: 16-byte units u0 .. u0+3 (u0 .. u0+1 under SwiGLU)
// of the lane's swizzled box row. Rows past M read no residual (the store
// clips them).
template <int EPI>
__device__ __forceinline__ void stage_chunk(const float (&v)[32], int row, int M, int col,
                                            const uint16_t* __restrict__ R, int ldc,
                                            uint8_t* box_row, int u0, int lane) {
  const int sw = lane & 7;
  auto put = [&](int u, uint4 w) {
    *reinterpret_cast<uint4*>(box_row + (((u0 + u) ^ sw) << 4)) = w;
  };
  if constexpr (EPI == GEMM_EPI_SWIGLU) {
    uint32_t o[8];
#pragma unroll
    for (int j = 0; j < 16; j += 2) {
      const float g0 = v[j], g1 = v[j + 1], u_0 = v[16 + j], u_1 = v[17 + j];
      o[j / 2] = pack_bf16(g0 / (1.f + expf(-g0)) * u_0, g1 / (1.f + expf(-g1)) * u_1);
    }
    put(0, make_uint4(o[0], o[1], o[2], o[3]));
    put(1, make_uint4(o[4], o[5], o[6], o[7]));
  } else {
    uint32_t o[16];
    if constexpr (EPI == GEMM_EPI_RESIDUAL) {
      const uint4* src = reinterpret_cast<const uint4*>(R + (int64_t)row * ldc + col);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 r4 = row < M ? src[q] : make_uint4(0, 0, 0, 0);
        const uint32_t rw[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int j = q * 8 + e * 2;
          o[q * 4 + e] = pack_bf16(v[j] + bf16_lo(rw[e]), v[j + 1] + bf16_hi(rw[e]));
        }
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; j += 2) o[j / 2] = pack_bf16(v[j], v[j + 1]);
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) put(q, make_uint4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]));
  }
}

// One epilogue warp's pass over its 32 rows of an accumulator: 8 chunks of
// 32 columns read with tcgen05.ld, staged into boxes, each full box stored
// by TMA. `nbox` counts the warp's boxes across tiles (it picks the buffer).
template <int EPI>
__device__ __forceinline__ void epilogue_rows(uint32_t t_row, int row0, int M, int col0,
                                              const uint16_t* __restrict__ R, int ldc,
                                              const CUtensorMap* map_c, uint8_t* boxes,
                                              int lane, int& nbox) {
  constexpr int CPB = epi_chunks_per_box<EPI>();
  constexpr int UPC = 8 / CPB;               // 16-byte units per chunk in a box row
#pragma unroll 1
  for (int c0 = 0; c0 < kBN; c0 += 32) {
    float v[32];
    tmem_ld32(t_row + c0, v);   // every lane takes part (.sync.aligned)
    const int cib = (c0 / 32) % CPB;
    uint8_t* box = boxes + (nbox & 1) * kEpiBox;
    if (cib == 0 && nbox >= 2) {   // the store that read this box two boxes ago
      if (lane == 0) epi_wait_read_1();
      __syncwarp();
    }
    stage_chunk<EPI>(v, row0 + lane, M, col0 + c0, R, ldc, box + lane * 128, cib * UPC, lane);
    if (cib == CPB - 1) {
      fence_async_smem();
      __syncwarp();
      if (lane == 0) {
        const int first = col0 + c0 - (CPB - 1) * 32;   // the box's first accumulator column
        const int x = EPI == GEMM_EPI_SWIGLU ? first / 2 : first;
        tma_store_2d(map_c, saddr(box), x, row0);
        epi_commit();
      }
      ++nbox;
    }
  }
}

// Persistent, warp-specialized: warp 0 loads (TMA), warp 1 issues the MMAs
// into one of two tensor-memory accumulators, warps 2..5 drain the other
// accumulator through the epilogue, so the epilogue of tile i overlaps the
// main loop of tile i + 1.
template <int EPI>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_bf16_kernel(const __grid_constant__ CUtensorMap map_a,
                     const __grid_constant__ CUtensorMap map_b,
                     const __grid_constant__ CUtensorMap map_c, int M, int N, int K,
                     const uint16_t* __restrict__ R, uint16_t* __restrict__ C, int ldc,
                     int* status) {
  extern __shared__ uint8_t gsm_raw[];
  // 1024-byte alignment: the 128-byte swizzle pattern repeats every 1024 bytes
  uint8_t* gsm = reinterpret_cast<uint8_t*>(((uintptr_t)gsm_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* epi_boxes = gsm + kStages * kStageBytes;   // [kEpiWarps][2] boxes, 1024-aligned
  uint64_t* full = reinterpret_cast<uint64_t*>(epi_boxes + kEpiSmem);
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;     // [2] accumulator ready (MMA -> epilogue)
  uint64_t* tempty = tfull + 2;          // [2] accumulator drained (epilogue -> MMA)
  uint64_t* done = tempty + 2;           // every issued MMA completed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  __shared__ int failed;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_m = (M + kBM - 1) / kBM, num_n = N / kBN;
  const int tiles = num_m * num_n;
  const int kt_n = K / kBK;

  if (threadIdx.x == 0) {
    failed = 0;
    for (int s = 0; s < kStages; ++s) {
      mbar_init(saddr(&full[s]), 1);
      mbar_init(saddr(&empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(saddr(&tfull[a]), 1);
      mbar_init(saddr(&tempty[a]), kEpiWarps);
    }
    mbar_init(saddr(done), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     saddr(tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  volatile int* vfailed = &failed;

  if (warp == 0) {
    if (lane == 0) {
      // producer: K-slices of every tile of this CTA into the ring
      int it = 0;
      for (int t = blockIdx.x; t < tiles && !*vfailed; t += gridDim.x) {
        int mt, nt;
        tile_coords<kGroupRows / kBM>(t, num_m, num_n, &mt, &nt);
        for (int kt = 0; kt < kt_n; ++kt, ++it) {
          const int s = it % kStages;
          if (it >= kStages && !mbar_wait(saddr(&empty[s]), ((it / kStages) - 1) & 1)) {
            *vfailed = 1;
            break;
          }
          if (*vfailed) break;
          const uint32_t a_dst = saddr(gsm + s * kStageBytes);
          mbar_expect_tx(saddr(&full[s]), kStageBytes);
          tma_load_2d(a_dst, &map_a, kt * kBK, mt * kBM, saddr(&full[s]));
          tma_load_2d(a_dst + kStageA, &map_b, kt * kBK, nt * kBN, saddr(&full[s]));
        }
      }
      // drain: the last issued slices must have landed before the CTA exits
      for (int j = it - kStages < 0 ? 0 : it - kStages; j < it; ++j)
        mbar_wait(saddr(&full[j % kStages]), (j / kStages) & 1);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // MMA issuer
      int it = 0, lt = 0;
      for (int t = blockIdx.x; t < tiles && !*vfailed; t += gridDim.x, ++lt) {
        const int acc = lt & 1;
        if (lt >= 2 && !mbar_wait(saddr(&tempty[acc]), ((lt >> 1) - 1) & 1)) {
          *vfailed = 1;
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t d_tmem = tmem + acc * kBN;
        bool ok = true;
        for (int kt = 0; kt < kt_n; ++kt, ++it) {
          const int s = it % kStages;
          if (!mbar_wait(saddr(&full[s]), (it / kStages) & 1) || *vfailed) {
            *vfailed = 1;
            ok = false;
            break;
          }
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          const uint32_t a_base = saddr(gsm + s * kStageBytes);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            umma_bf16(d_tmem, desc_k128(a_base + 32 * k), desc_k128(a_base + kStageA + 32 * k),
                      (kt > 0 || k > 0) ? 1u : 0u);
          umma_commit(saddr(&empty[s]));
        }
        if (!ok) break;
        umma_commit(saddr(&tfull[acc]));
      }
      umma_commit(saddr(done));   // arrives when every MMA issued above has completed
      mbar_wait(saddr(done), 0);
    }
  } else {
    // epilogue warps: warp w reads tensor-memory lanes 32 (w % 4) .. + 31
    const int q = warp & 3;
    uint8_t* boxes = epi_boxes + q * 2 * kEpiBox;
    int lt = 0, nbox = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++lt) {
      const int acc = lt & 1;
      const bool ok = mbar_wait(saddr(&tfull[acc]), (lt >> 1) & 1);
      if (!ok || *vfailed) {
        *vfailed = 1;
        break;
      }
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      int mt, nt;
      tile_coords<kGroupRows / kBM>(t, num_m, num_n, &mt, &nt);
      const uint32_t t_row = tmem + acc * kBN + ((uint32_t)(q * 32) << 16);
      epilogue_rows<EPI>(t_row, mt * kBM + q * 32, M, nt * kBN, R, ldc, &map_c, boxes, lane,
                         nbox);
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(saddr(&tempty[acc]));
    }
    if (lane == 0) epi_wait_all();   // the boxes are read before the CTA leaves
  }
  __syncthreads();
  if (*vfailed && threadIdx.x == 0) atomicCAS(status, 0, (int)SCONE_ERR_CUDA);
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols)
                 : "memory");
}

// ---------------------------------------------------------------- SM pairs
// The same GEMM on pairs of SMs (a 2-CTA cluster, tcgen05 cta_group::2): a
// pair computes a 256 x 256 tile. CTA r of the pair loads rows 128r..128r+127
// of the tile's A slice and of its B slice (16 + 16 KB per stage, so 6
// stages fit), both completing on the leader's (rank 0) full barrier; the
// leader's thread issues tcgen05.mma with M = 256, which reads both CTAs'
// halves and writes rows 128r.. of the accumulator into CTA r's tensor
// memory. Commits are multicast to both CTAs' barriers; both CTAs' epilogue
// warps release an accumulator on the leader's barrier. Per SM, a K-slice
// moves 32 KB instead of 48 KB for the same MMA work.
constexpr int kPStages = 6;
constexpr int kPairAccs = 2;                                 // accumulators per CTA
constexpr uint32_t kPairTmemCols = kPairAccs * kBN;
constexpr uint32_t kPStageHalf = 128 * kBK * 2;             // 16 KB: A or B half
constexpr uint32_t kPStageBytes = 2 * kPStageHalf;          // per CTA
constexpr size_t kPairSmem = (size_t)kPStages * kPStageBytes + 1024 + 256 + kEpiSmem;
constexpr uint32_t kIdescPair = (1u << 4) | (1u << 7) | (1u << 10) |
                                ((uint32_t)(kBN >> 3) << 17) | ((uint32_t)(256 >> 4) << 24);

__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, int x,
                                                 int y, uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::"
      "bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar_cluster)
      : "memory");
}
__device__ __forceinline__ void umma_bf16_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n"
      " setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(kIdescPair), "r"(accumulate)
      : "memory");
}
// Arrives on the barrier at this shared offset in both CTAs of the pair.
__device__ __forceinline__ void umma_commit_pair(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(bar),
      "h"((uint16_t)3)
      : "memory");
}
template <int EPI>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
    gemm_bf16_pair_kernel(const __grid_constant__ CUtensorMap map_a,
                          const __grid_constant__ CUtensorMap map_b,
                          const __grid_constant__ CUtensorMap map_c, int M, int N, int K,
                          const uint16_t* __restrict__ R, uint16_t* __restrict__ C, int ldc,
                          int* status) {
  extern __shared__ uint8_t gsm_raw[];
  uint8_t* gsm = reinterpret_cast<uint8_t*>(((uintptr_t)gsm_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* epi_boxes = gsm + kPStages * kPStageBytes;   // [kEpiWarps][2] boxes, 1024-aligned
  uint64_t* full = reinterpret_cast<uint64_t*>(epi_boxes + kEpiSmem);
  uint64_t* empty = full + kPStages;
  uint64_t* tfull = empty + kPStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* done = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  __shared__ int failed;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const bool leader = rank == 0;
  const int num_m = (M + 255) / 256, num_n = N / kBN;
  const int tiles = num_m * num_n;
  const int kt_n = K / kBK;
  const int pair = blockIdx.x >> 1, pairs = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    failed = 0;
    for (int i = 0; i < kPStages; ++i) {
      mbar_init(saddr(&full[i]), 1);
      mbar_init(saddr(&empty[i]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(saddr(&tfull[a]), 1);
      mbar_init(saddr(&tempty[a]), 2 * kEpiWarps);
    }
    mbar_init(saddr(done), 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     saddr(tmem_slot)),
                 "r"(kPairTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  cluster_sync();   // barriers initialized and tensor memory allocated in both CTAs
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  volatile int* vfailed = &failed;

  if (warp == 0) {
    if (lane == 0) {
      // producer (both CTAs): this CTA's halves, completing on the leader's full barrier
      int it = 0;
      for (int t = pair; t < tiles && !*vfailed; t += pairs) {
        int mt, nt;
        tile_coords<kGroupRows / 256>(t, num_m, num_n, &mt, &nt);
        for (int kt = 0; kt < kt_n; ++kt, ++it) {
          const int st = it % kPStages;
          if (it >= kPStages && !mbar_wait(saddr(&empty[st]), ((it / kPStages) - 1) & 1)) {
            *vfailed = 1;
            break;
          }
          if (*vfailed) break;
          const uint32_t a_dst = saddr(gsm + st * kPStageBytes);
          const uint32_t full_leader = map_to_rank(saddr(&full[st]), 0);
          if (leader) mbar_expect_tx(saddr(&full[st]), 2 * kPStageBytes);
          tma_load_2d_pair(a_dst, &map_a, kt * kBK, mt * 256 + (int)rank * 128, full_leader);
          tma_load_2d_pair(a_dst + kPStageHalf, &map_b, kt * kBK, nt * kBN + (int)rank * 128,
                           full_leader);
        }
      }
      if (leader)   // the last slices (both halves) must have landed before exit
        for (int j = it - kPStages < 0 ? 0 : it - kPStages; j < it; ++j)
          mbar_wait(saddr(&full[j % kPStages]), (j / kPStages) & 1);
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      int it = 0, lt = 0;
      for (int t = pair; t < tiles && !*vfailed; t += pairs, ++lt) {
        const int acc = lt % kPairAccs;
        if (lt >= kPairAccs && !mbar_wait(saddr(&tempty[acc]), ((lt / kPairAccs) - 1) & 1)) {
          *vfailed = 1;
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t d_tmem = tmem + acc * kBN;
        bool ok = true;
        for (int kt = 0; kt < kt_n; ++kt, ++it) {
          const int st = it % kPStages;
          if (!mbar_wait(saddr(&full[st]), (it / kPStages) & 1) || *vfailed) {
            *vfailed = 1;
            ok = false;
            break;
          }
          asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
          const uint32_t a_base = saddr(gsm + st * kPStageBytes);
#pragma unroll
          for (int k = 0; k < kBK / 16; ++k)
            umma_bf16_pair(d_tmem, desc_k128(a_base + 32 * k),
                           desc_k128(a_base + kPStageHalf + 32 * k), (kt > 0 || k > 0) ? 1u : 0u);
          umma_commit_pair(saddr(&empty[st]));
        }
        if (!ok) break;
        umma_commit_pair(saddr(&tfull[acc]));
      }
      umma_commit_pair(saddr(done));
    }
  } else {
    const int q = warp & 3;
    const uint32_t tempty_leader0 = map_to_rank(saddr(&tempty[0]), 0);
    const uint32_t tempty_leader1 = map_to_rank(saddr(&tempty[1]), 0);
    uint8_t* boxes = epi_boxes + q * 2 * kEpiBox;
    int lt = 0, nbox = 0;
    for (int t = pair; t < tiles; t += pairs, ++lt) {
      const int acc = lt % kPairAccs;
      if (!mbar_wait(saddr(&tfull[acc]), (lt / kPairAccs) & 1) || *vfailed) {
        *vfailed = 1;
        break;
      }
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      int mt, nt;
      tile_coords<kGroupRows / 256>(t, num_m, num_n, &mt, &nt);
      const uint32_t t_row = tmem + acc * kBN + ((uint32_t)(q * 32) << 16);
      epilogue_rows<EPI>(t_row, mt * 256 + (int)rank * 128 + q * 32, M, nt * kBN, R, ldc,
                         &map_c, boxes, lane, nbox);
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(acc ? tempty_leader1 : tempty_leader0);
    }
    if (lane == 0) epi_wait_all();   // the boxes are read before the CTA leaves
  }
  // every MMA of the pair has completed before either CTA frees its tensor memory
  if (threadIdx.x == 32) mbar_wait(saddr(done), 0);
  __syncthreads();
  if (*vfailed && threadIdx.x == 0) atomicCAS(status, 0, (int)SCONE_ERR_CUDA);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  cluster_sync();   // no CTA leaves while its peer may still signal its barriers
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kPairTmemCols)
                 : "memory");
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    else
      cudaGetLastError();
  });
  return fn;
}

// 2-D map of a row-major bf16 matrix [rows x cols] (cols contiguous), box
// 64 columns x box_rows rows, 128-byte swizzle; rows past the end read zero.
bool make_map(CUtensorMap* m, const void* base, int rows, int cols, int box_rows) {
  const auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kBK, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
         CUDA_SUCCESS;
}

// 2-D map of C [rows x ldc] for the epilogue's stores: box 64 columns x 32
// rows, 128-byte swizzle (as the boxes are staged); rows past the end are
// clipped.
bool make_map_c(CUtensorMap* m, void* base, int rows, int ldc) {
  const auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)ldc, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)ldc * 2};
  const cuuint32_t box[2] = {(cuuint32_t)kEpiBoxCols, 32};
  const cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int EPI>
bool set_smem_attr() {
  static std::once_flag once;
  static bool ok = false;
  std::call_once(once, [] {
    ok = cudaFuncSetAttribute(gemm_bf16_kernel<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)kGemmSmem) == cudaSuccess;
    if (!ok) cudaGetLastError();
  });
  return ok;
}

template <int EPI>
bool set_pair_smem_attr() {
  static std::once_flag once;
  static bool ok = false;
  std::call_once(once, [] {
    ok = cudaFuncSetAttribute(gemm_bf16_pair_kernel<EPI>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)kPairSmem) == cudaSuccess;
    if (!ok) cudaGetLastError();
  });
  return ok;
}

template <int EPI>
int launch_pair(const CUtensorMap& ma, const CUtensorMap& mb, int M, int N, int K,
                const uint16_t* R, uint16_t* C, int ldc, int* status, cudaStream_t s) {
  if (!set_pair_smem_attr<EPI>()) return SCONE_ERR_CUDA;
  CUtensorMap mc;
  if (!make_map_c(&mc, C, M, ldc)) return SCONE_ERR_CUDA;
  const int64_t tiles = (int64_t)((M + 255) / 256) * (N / kBN);
  const int64_t pairs = sm_count() / 2;
  const unsigned grid = (unsigned)(2 * (tiles < pairs ? tiles : pairs));
  gemm_bf16_pair_kernel<EPI><<<grid, kGemmThreads, kPairSmem, s>>>(ma, mb, mc, M, N, K, R, C,
                                                                   ldc, status);
  return cudaGetLastError() == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}

template <int EPI>
int launch_single(const CUtensorMap& ma, const CUtensorMap& mb, int M, int N, int K,
                  const uint16_t* R, uint16_t* C, int ldc, int* status, cudaStream_t s) {
  if (!set_smem_attr<EPI>()) return SCONE_ERR_CUDA;
  CUtensorMap mc;
  if (!make_map_c(&mc, C, M, ldc)) return SCONE_ERR_CUDA;
  const int64_t tiles = (int64_t)((M + kBM - 1) / kBM) * (N / kBN);
  const int64_t sms = sm_count();
  const dim3 grid((unsigned)(tiles < sms ? tiles : sms));
  gemm_bf16_kernel<EPI><<<grid, kGemmThreads, kGemmSmem, s>>>(ma, mb, mc, M, N, K, R, C, ldc,
                                                             status);
  return cudaGetLastError() == cudaSuccess ? SCONE_OK : SCONE_ERR_CUDA;
}

}  // namespace

int gemm_bf16(const uint16_t* A, const uint16_t* B, const uint16_t* R, uint16_t* C, int M, int N,
              int K, int epi, int* status, cudaStream_t s) {
  return gemm_bf16_variant(A, B, R, C, M, N, K, epi, 0, status, s);
}

int gemm_bf16_variant(const uint16_t* A, const uint16_t* B, const uint16_t* R, uint16_t* C,
                      int M, int N, int K, int epi, int variant, int* status, cudaStream_t s) {
  if (M < 0 || N <= 0 || K <= 0 || N % kBN || K % kBK || !A || !B || !C || !status)
    return SCONE_ERR_INVALID_ARG;
  if (epi == GEMM_EPI_RESIDUAL && !R) return SCONE_ERR_INVALID_ARG;
  if (((uintptr_t)A | (uintptr_t)B | (uintptr_t)C | (uintptr_t)R) & 15)
    return SCONE_ERR_INVALID_ARG;
  if (M == 0) return SCONE_OK;
  if (variant < 0 || variant > 2) return SCONE_ERR_INVALID_ARG;
  const int ldc = epi == GEMM_EPI_SWIGLU ? N / 2 : N;
  if (variant != 1) {   // SM pairs: 128-row halves of A and B per CTA
    CUtensorMap pa, pb;
    if (!make_map(&pa, A, M, K, 128) || !make_map(&pb, B, N, K, 128)) return SCONE_ERR_CUDA;
    switch (epi) {
      case GEMM_EPI_STORE:
        return launch_pair<GEMM_EPI_STORE>(pa, pb, M, N, K, R, C, ldc, status, s);
      case GEMM_EPI_RESIDUAL:
        return launch_pair<GEMM_EPI_RESIDUAL>(pa, pb, M, N, K, R, C, ldc, status, s);
      case GEMM_EPI_SWIGLU:
        return launch_pair<GEMM_EPI_SWIGLU>(pa, pb, M, N, K, R, C, ldc, status, s);
      default: return SCONE_ERR_INVALID_ARG;
    }
  }
  CUtensorMap ma, mb;
  if (!make_map(&ma, A, M, K, kBM) || !make_map(&mb, B, N, K, kBN)) return SCONE_ERR_CUDA;
  switch (epi) {
    case GEMM_EPI_STORE:
      return launch_single<GEMM_EPI_STORE>(ma, mb, M, N, K, R, C, ldc, status, s);
    case GEMM_EPI_RESIDUAL:
      return launch_single<GEMM_EPI_RESIDUAL>(ma, mb, M, N, K, R, C, ldc, status, s);
    case GEMM_EPI_SWIGLU:
      return launch_single<GEMM_EPI_SWIGLU>(ma, mb, M, N, K, R, C, ldc, status, s);
    default:
      return SCONE_ERR_INVALID_ARG;
  }
}

}  // namespace scone

extern "C" int scone_gemm_bf16(const scone_bf16* A, const scone_bf16* B, const scone_bf16* R,
                               scone_bf16* C, int32_t M, int32_t N, int32_t K, int32_t epilogue,
                               int* status, void* stream) {
  return scone::gemm_bf16(A, B, R, C, M, N, K, epilogue, status, (cudaStream_t)stream);
}

extern "C" int scone_gemm_bf16_variant(const scone_bf16* A, const scone_bf16* B,
                                       const scone_bf16* R, scone_bf16* C, int32_t M, int32_t N,
                                       int32_t K, int32_t epilogue, int32_t variant, int* status,
                                       void* stream) {
  return scone::gemm_bf16_variant(A, B, R, C, M, N, K, epilogue, variant, status,
                                  (cudaStream_t)stream);
}
