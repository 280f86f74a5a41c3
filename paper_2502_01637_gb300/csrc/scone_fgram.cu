// Precomputing F with the f-gram model (C ABI).
//
// At inference F(w) is the f-gram model's output for w, computed once and
// stored (Sec. 3.2; Algorithm 1 uses A_fgram(T(s_j), .., T(s_i)) in training
// and the stored F(s_j, .., s_i) at inference). The model is a pre-LN
// transformer: its input is the f-gram's token rows plus absolute position
// embeddings P[0..n-1] (Appendix F: an absolute position embedding layer
// with as many positions as the longest f-gram); per layer
// h = x + Attn(LN(x)), x = h + MLP(LN(h)), with non-parametric layer norm
// (eps 1e-5), causal multi-head attention and a SwiGLU MLP; F(w) is the layer
// norm of the last position's final state. Rotary positions on q and k
// (rotate-half pairs, base 10000) replace P when a model is created with
// SCONE_FGRAM_POS_ROTARY; that option is not the paper's scheme.
//
// Appendix F pads the f-grams of a batch to the longest one; the padding
// follows the last token and the attention is causal, so the last token's
// output does not depend on it, and the f-grams are packed here without it.
//
// The f-grams of a batch are packed token after token (no padding) into one
// [M x d] activation matrix, M = sum of their lengths, so every dense layer
// is one GEMM over all tokens of the batch on the tensor cores
// (scone_gemm.cu): qkv, the output projection with the residual added in
// its epilogue, gate/up with SwiGLU in its epilogue, and down with the
// residual. What is not a contraction runs on the CUDA cores, one warp per
// row or per (f-gram, head): the token-row gather, layer norm, attention over
// at most K positions, and the final layer norm written to F.

#include <cuda_bf16.h>

#include <new>
#include <type_traits>

#include "scone_gemm.h"
#include "scone_host.h"

struct scone_fgram_model {
  int device = 0;
  int32_t d = 0, n_heads = 0, ffw = 0, n_layers = 0;
  int32_t max_pos = 0;                   // rows of P (absolute positions)
  int32_t position = 0;                  // SCONE_FGRAM_POS_ABSOLUTE or _ROTARY
  const uint16_t* weights = nullptr;     // borrowed, packed layout
  const uint16_t* P = nullptr;           // [max_pos x d] inside weights; null for rotary
  int64_t batch = 0;                     // f-grams per batch
  int64_t cap_rows = 0;                  // workspace rows (tokens)
  int32_t* off = nullptr;                // [batch + 1] token offsets
  int* status = nullptr;                 // sticky device error
  int* h_words = nullptr;                // pinned [2]: a batch's token count, the status
  uint16_t *X = nullptr, *Xn = nullptr, *QKV = nullptr, *Act = nullptr;
};

namespace scone {

namespace {

constexpr float kLnEps = 1e-5f;
constexpr int kRowsPerBlock = 8;       // one warp per row, 8 warps per block

__device__ __forceinline__ void set_error(int* status, int code) {
  if (*reinterpret_cast<volatile int*>(status) == 0) atomicCAS(status, 0, code);
}

__device__ __forceinline__ float lo_f(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float hi_f(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t pack2(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// Exclusive prefix sum of the batch's lengths (one block): off[0..n].
__global__ void __launch_bounds__(1024)
    offsets_kernel(const uint8_t* __restrict__ len, int64_t n, int32_t K, int32_t* __restrict__ off,
                   int* status) {
  __shared__ int32_t part[1024];
  const int64_t per = (n + 1023) / 1024;
  const int64_t b = threadIdx.x * per, e = b + per < n ? b + per : n;
  int32_t s = 0;
  for (int64_t i = b; i < e; ++i) {
    int32_t l = len[i];
    if (l < 1 || l > K) {
      set_error(status, SCONE_ERR_INVALID_ARG);
      l = 1;
    }
    s += l;
  }
  part[threadIdx.x] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    int32_t run = 0;
    for (int t = 0; t < 1024; ++t) {
      const int32_t v = part[t];
      part[t] = run;
      run += v;
    }
    off[n] = run;
  }
  __syncthreads();
  int32_t run = part[threadIdx.x];
  for (int64_t i = b; i < e; ++i) {
    off[i] = run;
    int32_t l = len[i];
    run += (l < 1 || l > K) ? 1 : l;
  }
}

__device__ __forceinline__ uint32_t add2(uint32_t a, uint32_t b) {
  return pack2(lo_f(a) + lo_f(b), hi_f(a) + hi_f(b));
}

// The model input: X[off[f] + j] = bf16(T[tok[f * K + j]] + P[j]) (fp32 sum,
// rounded to nearest even), or T's row alone when P is null; one warp per
// f-gram. Position j counts from the f-gram's first token; j < K <= max_pos
// is checked on the host, and rows past a length outside [1, K] are not
// read (offsets_kernel counts such an f-gram as one token).
__global__ void __launch_bounds__(256)
    gather_rows_kernel(const int32_t* __restrict__ tok, const uint8_t* __restrict__ len,
                       const int32_t* __restrict__ off, int64_t n, int32_t K,
                       const uint16_t* __restrict__ T, int32_t vocab, int32_t d,
                       const uint16_t* __restrict__ P, uint16_t* __restrict__ X, int* status) {
  const int lane = threadIdx.x & 31;
  const int64_t f = (int64_t)blockIdx.x * kRowsPerBlock + (threadIdx.x >> 5);
  if (f >= n) return;
  const int nl = off[f + 1] - off[f];
  const int chunks = d / 8;                       // 16-byte chunks per row
  for (int j = 0; j < nl; ++j) {
    const int32_t t = tok[f * K + j];
    uint4* dst = reinterpret_cast<uint4*>(X + (int64_t)(off[f] + j) * d);
    if ((uint32_t)t >= (uint32_t)vocab) {
      if (lane == 0) set_error(status, SCONE_ERR_TOKEN_RANGE);
      for (int c = lane; c < chunks; c += 32) dst[c] = make_uint4(0, 0, 0, 0);
      continue;
    }
    const uint4* src = reinterpret_cast<const uint4*>(T + (int64_t)t * d);
    if (!P) {
      for (int c = lane; c < chunks; c += 32) dst[c] = __ldg(src + c);
      continue;
    }
    const uint4* pos = reinterpret_cast<const uint4*>(P + (int64_t)j * d);
    for (int c = lane; c < chunks; c += 32) {
      const uint4 a = __ldg(src + c), b = __ldg(pos + c);
      dst[c] = make_uint4(add2(a.x, b.x), add2(a.y, b.y), add2(a.z, b.z), add2(a.w, b.w));
    }
  }
}

// Non-parametric layer norm of rows (one warp per row): Y = (X - mean) /
// sqrt(var + eps), CH = d / 256 16-byte chunks per lane. With `off`, output
// row r is the layer norm of input row off[r + 1] - 1, the last position of
// f-gram r (the F rows).
template <int CH>
__global__ void __launch_bounds__(256)
    layernorm_kernel(const uint16_t* __restrict__ X, uint16_t* __restrict__ Y, int64_t n_rows,
                     const int32_t* __restrict__ off) {
  const int lane = threadIdx.x & 31;
  const int64_t r = (int64_t)blockIdx.x * kRowsPerBlock + (threadIdx.x >> 5);
  if (r >= n_rows) return;
  constexpr int d = CH * 256;
  const int64_t src_row = off ? (int64_t)off[r + 1] - 1 : r;   // last position of f-gram r
  const uint4* src = reinterpret_cast<const uint4*>(X + src_row * d);
  float v[CH * 8];
  float sum = 0.f;
#pragma unroll
  for (int c = 0; c < CH; ++c) {
    const uint4 q = __ldg(src + c * 32 + lane);
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      v[c * 8 + 2 * e] = lo_f(w[e]);
      v[c * 8 + 2 * e + 1] = hi_f(w[e]);
      sum += v[c * 8 + 2 * e] + v[c * 8 + 2 * e + 1];
    }
  }
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
  const float mean = sum / d;
  float sq = 0.f;
#pragma unroll
  for (int i = 0; i < CH * 8; ++i) {
    v[i] -= mean;
    sq += v[i] * v[i];
  }
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xFFFFFFFFu, sq, o);
  const float inv = rsqrtf(sq / d + kLnEps);
  uint4* dst = reinterpret_cast<uint4*>(Y + r * d);
#pragma unroll
  for (int c = 0; c < CH; ++c) {
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) w[e] = pack2(v[c * 8 + 2 * e] * inv, v[c * 8 + 2 * e + 1] * inv);
    dst[c * 32 + lane] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

// C consecutive bf16 moved as one 2-, 4- or 8-byte word.
template <int C>
struct Lanes {
  using Word = typename std::conditional<C == 1, uint16_t,
                                         typename std::conditional<C == 2, uint32_t,
                                                                   uint2>::type>::type;
  union {
    Word w;
    uint16_t h[C];
  } u;
  __device__ __forceinline__ static Lanes load(const uint16_t* p) {
    Lanes x;
    x.u.w = __ldg(reinterpret_cast<const Word*>(p));
    return x;
  }
  __device__ __forceinline__ float get(int e) const {
    return __uint_as_float((uint32_t)u.h[e] << 16);
  }
  __device__ __forceinline__ void set(int e, float f) {
    const __nv_bfloat16 b = __float2bfloat16_rn(f);
    u.h[e] = *reinterpret_cast<const uint16_t*>(&b);
  }
  __device__ __forceinline__ void store(uint16_t* p) const {
    *reinterpret_cast<Word*>(p) = u.w;
  }
};

// Causal attention of one (f-gram, head) per warp over at most KMAX
// positions. Lane l holds dims C*l .. C*l+C-1 of the head's first half and the
// same offsets of its second half (C = hd / 64), so each rotate-half pair of
// the rotary embedding (applied when ROTARY) stays in one lane.
template <int C, int KMAX, bool ROTARY>
__global__ void __launch_bounds__(256)
    attention_kernel(const uint16_t* __restrict__ QKV, const int32_t* __restrict__ off, int64_t n,
                     int32_t d, int32_t H, uint16_t* __restrict__ O) {
  constexpr int hd = 64 * C, half = 32 * C;
  const int lane = threadIdx.x & 31;
  const int64_t wid = (int64_t)blockIdx.x * kRowsPerBlock + (threadIdx.x >> 5);
  if (wid >= n * H) return;
  const int64_t f = wid / H;
  const int h = (int)(wid % H);
  const int32_t r0 = off[f];
  const int nl = off[f + 1] - r0 < KMAX ? off[f + 1] - r0 : KMAX;
  float q[KMAX][2 * C], k[KMAX][2 * C], v[KMAX][2 * C];
  float theta[C];
#pragma unroll
  for (int e = 0; e < C; ++e)
    theta[e] = ROTARY ? powf(10000.f, -2.f * (float)(C * lane + e) / (float)hd) : 0.f;
#pragma unroll
  for (int j = 0; j < KMAX; ++j) {
    if (j >= nl) break;
    const uint16_t* row = QKV + (int64_t)(r0 + j) * 3 * d + h * hd;
#pragma unroll
    for (int part = 0; part < 2; ++part) {
      const int base = part * half + C * lane;
      const Lanes<C> a = Lanes<C>::load(row + base);
      const Lanes<C> b = Lanes<C>::load(row + d + base);
      const Lanes<C> c = Lanes<C>::load(row + 2 * d + base);
#pragma unroll
      for (int e = 0; e < C; ++e) {
        q[j][part * C + e] = a.get(e);
        k[j][part * C + e] = b.get(e);
        v[j][part * C + e] = c.get(e);
      }
    }
    // rotary embedding at position j: (a, b) -> (a cos - b sin, b cos + a sin)
#pragma unroll
    for (int e = 0; e < (ROTARY ? C : 0); ++e) {
      float s, c;
      sincosf((float)j * theta[e], &s, &c);
      const float qa = q[j][e], qb = q[j][C + e], ka = k[j][e], kb = k[j][C + e];
      q[j][e] = qa * c - qb * s;
      q[j][C + e] = qb * c + qa * s;
      k[j][e] = ka * c - kb * s;
      k[j][C + e] = kb * c + ka * s;
    }
  }
  const float scale = rsqrtf((float)hd);
#pragma unroll
  for (int i = 0; i < KMAX; ++i) {
    if (i >= nl) break;
    float sc[KMAX];
    float mx = -INFINITY;
#pragma unroll
    for (int j = 0; j < KMAX; ++j) {
      if (j > i) break;
      float p = 0.f;
#pragma unroll
      for (int e = 0; e < 2 * C; ++e) p += q[i][e] * k[j][e];
      for (int o = 16; o > 0; o >>= 1) p += __shfl_xor_sync(0xFFFFFFFFu, p, o);
      sc[j] = p * scale;
      mx = fmaxf(mx, sc[j]);
    }
    float den = 0.f, acc[2 * C];
#pragma unroll
    for (int e = 0; e < 2 * C; ++e) acc[e] = 0.f;
#pragma unroll
    for (int j = 0; j < KMAX; ++j) {
      if (j > i) break;
      const float p = expf(sc[j] - mx);
      den += p;
#pragma unroll
      for (int e = 0; e < 2 * C; ++e) acc[e] += p * v[j][e];
    }
    const float inv = 1.f / den;
    uint16_t* out = O + (int64_t)(r0 + i) * d + h * hd;
#pragma unroll
    for (int part = 0; part < 2; ++part) {
      Lanes<C> o;
#pragma unroll
      for (int e = 0; e < C; ++e) o.set(e, acc[part * C + e] * inv);
      o.store(out + part * half + C * lane);
    }
  }
}

template <int CH>
void launch_ln(const uint16_t* X, uint16_t* Y, int64_t rows, const int32_t* off,
               cudaStream_t s) {
  const unsigned grid = (unsigned)((rows + kRowsPerBlock - 1) / kRowsPerBlock);
  layernorm_kernel<CH><<<grid, 256, 0, s>>>(X, Y, rows, off);
}

bool ln(int d, const uint16_t* X, uint16_t* Y, int64_t rows, const int32_t* off, cudaStream_t s) {
  switch (d / 256) {
    case 1: launch_ln<1>(X, Y, rows, off, s); return true;
    case 2: launch_ln<2>(X, Y, rows, off, s); return true;
    case 4: launch_ln<4>(X, Y, rows, off, s); return true;
    case 8: launch_ln<8>(X, Y, rows, off, s); return true;
    case 16: launch_ln<16>(X, Y, rows, off, s); return true;
    default: return false;
  }
}

template <int KMAX, bool ROTARY>
bool attn_k(int hd, const uint16_t* QKV, const int32_t* off, int64_t n, int d, int H,
            uint16_t* O, cudaStream_t s) {
  const unsigned grid = (unsigned)((n * H + kRowsPerBlock - 1) / kRowsPerBlock);
  switch (hd) {
    case 64:
      attention_kernel<1, KMAX, ROTARY><<<grid, 256, 0, s>>>(QKV, off, n, d, H, O);
      return true;
    case 128:
      attention_kernel<2, KMAX, ROTARY><<<grid, 256, 0, s>>>(QKV, off, n, d, H, O);
      return true;
    case 256:
      attention_kernel<4, KMAX, ROTARY><<<grid, 256, 0, s>>>(QKV, off, n, d, H, O);
      return true;
    default: return false;
  }
}

// Positions held in registers: the smallest of 3, 5, 8 that covers K.
template <bool ROTARY>
bool attn_r(int K, int hd, const uint16_t* QKV, const int32_t* off, int64_t n, int d, int H,
            uint16_t* O, cudaStream_t s) {
  if (K <= 3) return attn_k<3, ROTARY>(hd, QKV, off, n, d, H, O, s);
  if (K <= 5) return attn_k<5, ROTARY>(hd, QKV, off, n, d, H, O, s);
  return attn_k<8, ROTARY>(hd, QKV, off, n, d, H, O, s);
}

bool attn(bool rotary, int K, int hd, const uint16_t* QKV, const int32_t* off, int64_t n, int d,
          int H, uint16_t* O, cudaStream_t s) {
  return rotary ? attn_r<true>(K, hd, QKV, off, n, d, H, O, s)
                : attn_r<false>(K, hd, QKV, off, n, d, H, O, s);
}

bool ensure_rows(scone_fgram_model* m, int64_t rows) {
  if (rows <= m->cap_rows) return true;
  for (uint16_t** p : {&m->X, &m->Xn, &m->QKV, &m->Act}) {
    if (*p) cudaFree(*p);
    *p = nullptr;
  }
  m->cap_rows = 0;
  const int64_t r = rows + rows / 8;
  if (cudaMalloc(&m->X, (size_t)r * m->d * 2) != cudaSuccess ||
      cudaMalloc(&m->Xn, (size_t)r * m->d * 2) != cudaSuccess ||
      cudaMalloc(&m->QKV, (size_t)r * 3 * m->d * 2) != cudaSuccess ||
      cudaMalloc(&m->Act, (size_t)r * m->ffw * 2) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  m->cap_rows = r;
  return true;
}

}  // namespace

}  // namespace scone

using namespace scone;

extern "C" int scone_fgram_model_create(int32_t d, int32_t n_heads, int32_t ffw, int32_t n_layers,
                                        int32_t max_pos, int32_t position,
                                        const scone_bf16* weights, int64_t batch,
                                        scone_fgram_model** out) {
  if (!out) return SCONE_ERR_INVALID_ARG;
  *out = nullptr;
  const bool absolute = position == SCONE_FGRAM_POS_ABSOLUTE;
  if (!absolute && position != SCONE_FGRAM_POS_ROTARY) return SCONE_ERR_INVALID_ARG;
  if (d <= 0 || d % 256 || d / 256 > 16 || (d / 256) & (d / 256 - 1) || n_heads <= 0 ||
      d % n_heads || ffw <= 0 || ffw % 128 || n_layers < 0 ||
      ((n_layers > 0 || absolute) && !weights) || ((uintptr_t)weights & 15) || batch < 0 ||
      (absolute && (max_pos < 1 || max_pos > 8)))
    return SCONE_ERR_INVALID_ARG;
  const int hd = d / n_heads;
  if (hd != 64 && hd != 128 && hd != 256) return SCONE_ERR_UNSUPPORTED;
  auto* m = new (std::nothrow) scone_fgram_model();
  if (!m) return SCONE_ERR_NOMEM;
  cudaGetDevice(&m->device);
  m->d = d;
  m->n_heads = n_heads;
  m->ffw = ffw;
  m->n_layers = n_layers;
  m->weights = weights;
  m->position = position;
  m->max_pos = absolute ? max_pos : 0;
  // P follows the last layer in the packed buffer
  const int64_t layer_elems = (int64_t)3 * d * d + (int64_t)d * d + (int64_t)2 * ffw * d +
                              (int64_t)d * ffw;
  m->P = absolute ? weights + n_layers * layer_elems : nullptr;
  m->batch = batch > 0 ? batch : 16384;
  if (cudaMalloc(&m->off, (size_t)(m->batch + 1) * sizeof(int32_t)) != cudaSuccess ||
      cudaMalloc(&m->status, sizeof(int)) != cudaSuccess ||
      cudaMemset(m->status, 0, sizeof(int)) != cudaSuccess ||
      cudaHostAlloc(&m->h_words, 2 * sizeof(int), cudaHostAllocDefault) != cudaSuccess) {
    cudaGetLastError();
    scone_fgram_model_destroy(m);
    return SCONE_ERR_NOMEM;
  }
  *out = m;
  return SCONE_OK;
}

extern "C" int scone_fgram_model_destroy(scone_fgram_model* m) {
  if (!m) return SCONE_OK;
  DeviceGuard g(m->device);
  cudaDeviceSynchronize();
  for (void* p : {(void*)m->off, (void*)m->status, (void*)m->X, (void*)m->Xn, (void*)m->QKV,
                  (void*)m->Act})
    if (p) cudaFree(p);
  if (m->h_words) cudaFreeHost(m->h_words);
  delete m;
  return SCONE_OK;
}

extern "C" int scone_fgram_precompute(scone_fgram_model* m, const int32_t* fgram_tok,
                                      const uint8_t* fgram_len, int64_t n, int32_t K,
                                      const scone_bf16* T, int32_t vocab, scone_bf16* F,
                                      void* stream) {
  if (!m || n < 0 || K < 2 || K > 8 || vocab < 1) return SCONE_ERR_INVALID_ARG;
  // every position of an f-gram needs a row of P
  if (m->position == SCONE_FGRAM_POS_ABSOLUTE && K > m->max_pos) return SCONE_ERR_INVALID_ARG;
  if (n == 0) return SCONE_OK;
  if (!fgram_tok || !fgram_len || !T || !F || ((uintptr_t)T & 15) || ((uintptr_t)F & 15) ||
      ((uintptr_t)fgram_tok & 3))
    return SCONE_ERR_INVALID_ARG;
  DeviceGuard g(m->device);
  cudaStream_t s = (cudaStream_t)stream;
  const int d = m->d, H = m->n_heads, ffw = m->ffw;
  const int64_t layer_elems = (int64_t)3 * d * d + (int64_t)d * d + (int64_t)2 * ffw * d +
                              (int64_t)d * ffw;
  for (int64_t f0 = 0; f0 < n; f0 += m->batch) {
    const int64_t nb = n - f0 < m->batch ? n - f0 : m->batch;
    offsets_kernel<<<1, 1024, 0, s>>>(fgram_len + f0, nb, K, m->off, m->status);
    if (cudaGetLastError() != cudaSuccess ||
        cudaMemcpyAsync(m->h_words, m->off + nb, sizeof(int32_t), cudaMemcpyDeviceToHost, s) !=
            cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
      return SCONE_ERR_CUDA;
    const int32_t rows = m->h_words[0];
    if (!ensure_rows(m, rows)) return SCONE_ERR_NOMEM;
    const unsigned gw = (unsigned)((nb + kRowsPerBlock - 1) / kRowsPerBlock);
    gather_rows_kernel<<<gw, 256, 0, s>>>(fgram_tok + f0 * K, fgram_len + f0, m->off, nb, K, T,
                                          vocab, d, m->P, m->X, m->status);
    for (int l = 0; l < m->n_layers; ++l) {
      const uint16_t* w = m->weights + l * layer_elems;
      const uint16_t* wqkv = w;
      const uint16_t* wo = wqkv + (int64_t)3 * d * d;
      const uint16_t* wgu = wo + (int64_t)d * d;
      const uint16_t* wd = wgu + (int64_t)2 * ffw * d;
      int rc;
      if (!ln(d, m->X, m->Xn, rows, nullptr, s)) return SCONE_ERR_UNSUPPORTED;
      if ((rc = gemm_bf16(m->Xn, wqkv, nullptr, m->QKV, rows, 3 * d, d, GEMM_EPI_STORE,
                          m->status, s)))
        return rc;
      if (!attn(m->position == SCONE_FGRAM_POS_ROTARY, K, d / H, m->QKV, m->off, nb, d, H,
                m->Xn, s))
        return SCONE_ERR_UNSUPPORTED;
      if ((rc = gemm_bf16(m->Xn, wo, m->X, m->X, rows, d, d, GEMM_EPI_RESIDUAL, m->status, s)))
        return rc;
      if (!ln(d, m->X, m->Xn, rows, nullptr, s)) return SCONE_ERR_UNSUPPORTED;
      if ((rc = gemm_bf16(m->Xn, wgu, nullptr, m->Act, rows, 2 * ffw, d, GEMM_EPI_SWIGLU,
                          m->status, s)))
        return rc;
      if ((rc = gemm_bf16(m->Act, wd, m->X, m->X, rows, d, ffw, GEMM_EPI_RESIDUAL, m->status,
                          s)))
        return rc;
    }
    // F rows: layer norm of each f-gram's last position
    if (!ln(d, m->X, F + f0 * d, nb, m->off, s)) return SCONE_ERR_UNSUPPORTED;
    if (cudaGetLastError() != cudaSuccess) return SCONE_ERR_CUDA;
  }
  if (cudaMemcpyAsync(m->h_words + 1, m->status, sizeof(int), cudaMemcpyDeviceToHost, s) !=
          cudaSuccess ||
      cudaMemsetAsync(m->status, 0, sizeof(int), s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return SCONE_ERR_CUDA;
  return m->h_words[1];
}
