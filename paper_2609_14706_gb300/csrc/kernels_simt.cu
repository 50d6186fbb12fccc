// CUDA-core kernels of the FlipFlop Hessian fit:
//  * blocked right-looking Cholesky (fp32): 64 x 64 diagonal blocks factored and
//    inverted in shared memory by one CTA, panel TRSM and trailing SYRK as tiled GEMMs;
//  * triangular inverse M = L^-1 by recursive doubling: with the 64 x 64 diagonal
//    inverses known, [[L11,0],[L21,L22]]^-1 has off-diagonal block -M22 (L21 M11),
//    two batched GEMMs per level;
//  * conversions, the A_0 = I shortcut q_k = ||x_k||^2, damping, trace normalisation,
//    the convergence statistics and fp64 dot products;
//  * CUDA-core versions of the weighted Gram and the quadratic form (option kernel=1),
//    used to cross-check the tensor-core kernels.
#include <algorithm>
#include <atomic>

#include "ffh_internal.cuh"

namespace ffh {

static std::atomic<long long> g_launches{0};
void note_launches(int k) { g_launches.fetch_add(k, std::memory_order_relaxed); }
long long launches_so_far() { return g_launches.load(std::memory_order_relaxed); }

// SM count of the current device (cached per device; read and written atomically)
int num_sms() {
  static std::atomic<int> cache[64];
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c > 0) return c;
  }
  int sms = 0;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (sms <= 0) sms = 1;
  if (dev >= 0 && dev < 64) cache[dev].store(sms, std::memory_order_relaxed);
  return sms;
}

template <typename T>
__device__ __forceinline__ float ldf(const T* p);
template <>
__device__ __forceinline__ float ldf<float>(const float* p) {
  return *p;
}
template <>
__device__ __forceinline__ float ldf<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}

__device__ __forceinline__ double block_sum_f64(double v) {
  __shared__ double red[32];
  for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  v = 0.0;
  if (w == 0) {
    const int nw = (blockDim.x + 31) >> 5;
    v = l < nw ? red[l] : 0.0;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
  }
  return v;  // valid in thread 0
}

// ---------------------------------------------------------------------------
// row sums of squares: q_k = ||v_k||^2 (first B-update, A_0 = I)
// ---------------------------------------------------------------------------
template <typename T>
__global__ void k_rowsumsq(const T* __restrict__ V, int64_t N, int64_t d, int64_t ld,
                           float* __restrict__ q) {
  const int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= N) return;
  const T* v = V + row * ld;
  float acc = 0.f;
  for (int64_t j = lane; j < d; j += 32) {
    const float x = ldf(v + j);
    acc = fmaf(x, x, acc);
  }
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, o);
  if (lane == 0) q[row] = acc;
}

cudaError_t launch_rowsumsq(const void* V, int dtype, int64_t N, int64_t d, int64_t ld, float* q,
                            cudaStream_t s) {
  const int wpb = 8;
  const int64_t blocks = (N + wpb - 1) / wpb;
  if (blocks == 0) return cudaSuccess;
  if (dtype == FFH_BF16) {
    k_rowsumsq<<<(unsigned)blocks, wpb * 32, 0, s>>>(static_cast<const __nv_bfloat16*>(V), N, d,
                                                      ld, q);
  } else {
    k_rowsumsq<<<(unsigned)blocks, wpb * 32, 0, s>>>(static_cast<const float*>(V), N, d, ld, q);
  }
  note_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// fp32 -> bf16 (pitch change, zero padding; `lower`: zero the strict upper triangle)
// ---------------------------------------------------------------------------
__global__ void k_to_bf16(const float* __restrict__ src, int64_t rows, int64_t cols, int64_t lds,
                          __nv_bfloat16* __restrict__ dst, int64_t ldd, int lower) {
  const int64_t total = rows * ldd;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = idx / ldd, c = idx - r * ldd;
    float v = 0.f;
    if (c < cols && !(lower && c > r)) v = src[r * lds + c];
    dst[idx] = __float2bfloat16_rn(v);
  }
}

cudaError_t launch_to_bf16_ex(const float* src, int64_t rows, int64_t cols, int64_t lds,
                              __nv_bfloat16* dst, int64_t ldd, int lower, cudaStream_t s) {
  const int64_t total = rows * ldd;
  if (total == 0) return cudaSuccess;
  const int64_t blocks = std::min<int64_t>((total + 255) / 256, (int64_t)num_sms() * 32);
  k_to_bf16<<<(unsigned)blocks, 256, 0, s>>>(src, rows, cols, lds, dst, ldd, lower); note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_to_bf16(const float* src, int64_t rows, int64_t cols, int64_t lds,
                           __nv_bfloat16* dst, int64_t ldd, cudaStream_t s) {
  return launch_to_bf16_ex(src, rows, cols, lds, dst, ldd, 0, s);
}

cudaError_t launch_lower_to_bf16(const float* src, int64_t d, int64_t lds, __nv_bfloat16* dst,
                                 int64_t ldd, cudaStream_t s) {
  return launch_to_bf16_ex(src, d, d, lds, dst, ldd, 1, s);
}

// dst[r][c] = src[c][r] for c >= r (the transpose of a lower-triangular src), 0 below;
// 32 x 32 tiles through shared memory
__global__ void k_lowerT_to_bf16(const float* __restrict__ src, int64_t d, int64_t lds,
                                 __nv_bfloat16* __restrict__ dst, int64_t ldd) {
  __shared__ float t[32][33];
  const int64_t bx = (int64_t)blockIdx.x * 32, by = (int64_t)blockIdx.y * 32;
  for (int r = threadIdx.y; r < 32; r += 8) {
    const int64_t sr = by + r, sc = bx + threadIdx.x;  // source row sr, column sc
    t[r][threadIdx.x] = (sr < d && sc < d && sc <= sr) ? src[sr * lds + sc] : 0.f;
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += 8) {
    const int64_t dr = bx + r, dc = by + threadIdx.x;  // dst row = source column
    if (dr < ldd && dc < ldd && dr < d + 8) {
      if (dr < d) dst[dr * ldd + dc] = __float2bfloat16_rn(dc < d ? t[threadIdx.x][r] : 0.f);
    }
  }
}

cudaError_t launch_lowerT_to_bf16(const float* src, int64_t d, int64_t lds, __nv_bfloat16* dst,
                                  int64_t ldd, cudaStream_t s) {
  const unsigned nb = (unsigned)((ldd + 31) / 32);
  k_lowerT_to_bf16<<<dim3(nb, nb), dim3(32, 8), 0, s>>>(src, d, lds, dst, ldd);
  note_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// tiled fp32 GEMM (64 x 64 tiles, 256 threads, 4 x 4 per thread), batched over z:
//   C = alpha * A * op(B) + beta * C,  op(B) = B (K x N) or B^T (B is N x K)
// with triangular skips:
//   LOWER_C     tiles strictly above the diagonal are skipped
//   A_LOWER     A[r][k] = 0 for k > r  (K range ends at the tile's last row)
//   B_LOWER_NN  B[k][c] = 0 for k < c  (K range starts at the tile's first column)
//   B_LOWER_NT  op(B)[k][c] = B[c][k] = 0 for k > c (K range ends at its last column)
// ---------------------------------------------------------------------------
enum { GF_LOWER_C = 1, GF_A_LOWER = 2, GF_B_LOWER_NN = 4, GF_B_LOWER_NT = 8, GF_TRANS_B = 16 };

struct GemmArgs {
  const float* A;
  int64_t lda, strideA;
  const float* B;
  int64_t ldb, strideB;
  float* C;
  int64_t ldc, strideC;
  int M, N, K;
  float alpha, beta;
  int flags;
};

__global__ void __launch_bounds__(256) k_gemm64(const GemmArgs g) {
  const int row0 = blockIdx.y * 64, col0 = blockIdx.x * 64;
  if ((g.flags & GF_LOWER_C) && col0 > row0 + 63) return;
  const int z = blockIdx.z;
  const float* A = g.A + (int64_t)z * g.strideA;
  const float* B = g.B + (int64_t)z * g.strideB;
  float* C = g.C + (int64_t)z * g.strideC;
  int k_lo = 0, k_hi = g.K;
  if (g.flags & GF_A_LOWER) k_hi = min(k_hi, row0 + 64);
  if (g.flags & GF_B_LOWER_NT) k_hi = min(k_hi, col0 + 64);
  if (g.flags & GF_B_LOWER_NN) k_lo = col0 & ~15;
  const bool transB = (g.flags & GF_TRANS_B) != 0;

  __shared__ float As[16][68];
  __shared__ float Bs[16][68];
  const int tid = threadIdx.x;
  const int ty = tid >> 4, tx = tid & 15;
  float acc[4][4] = {};
  for (int k0 = k_lo; k0 < k_hi; k0 += 16) {
    // A tile: 64 rows x 16 k (each thread 4 elements, k fastest for coalescing)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int idx = tid + e * 256;
      const int r = idx >> 4, kk = idx & 15;
      const int gr = row0 + r, gk = k0 + kk;
      As[kk][r] = (gr < g.M && gk < k_hi) ? A[(int64_t)gr * g.lda + gk] : 0.f;
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int idx = tid + e * 256;
      if (!transB) {
        const int kk = idx >> 6, c = idx & 63;
        const int gk = k0 + kk, gc = col0 + c;
        Bs[kk][c] = (gk < k_hi && gc < g.N) ? B[(int64_t)gk * g.ldb + gc] : 0.f;
      } else {
        const int c = idx >> 4, kk = idx & 15;
        const int gk = k0 + kk, gc = col0 + c;
        Bs[kk][c] = (gk < k_hi && gc < g.N) ? B[(int64_t)gc * g.ldb + gk] : 0.f;
      }
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int gr = row0 + ty * 4 + i;
    if (gr >= g.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int gc = col0 + tx * 4 + j;
      if (gc >= g.N) continue;
      float* cp = C + (int64_t)gr * g.ldc + gc;
      const float v = g.alpha * acc[i][j];
      *cp = (g.beta == 0.f) ? v : fmaf(g.beta, *cp, v);
    }
  }
}

static cudaError_t gemm(const GemmArgs& g, int batch, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0 || batch <= 0) return cudaSuccess;
  dim3 grid((g.N + 63) / 64, (g.M + 63) / 64, batch);
  k_gemm64<<<grid, 256, 0, s>>>(g); note_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Cholesky
// ---------------------------------------------------------------------------
constexpr int NB = 64;

// Factor the (already updated) diagonal block p of W in shared memory, write its
// Cholesky factor into L and its inverse into DI (64 x 64), accumulate log|.|.
__global__ void __launch_bounds__(256) k_chol_diag(float* W, int64_t ldw, int64_t d, int p,
                                                   float* L, int64_t ldl, float* DI,
                                                   DevStatus* st, int fault) {
  __shared__ float s[NB][NB + 1];
  __shared__ float inv[NB][NB + 1];
  __shared__ double ld_acc;
  __shared__ int bad;
  const int64_t o = (int64_t)p * NB;
  const int b = (int)((d - o) < NB ? (d - o) : NB);
  const int tid = threadIdx.x;
  if (tid == 0) {
    ld_acc = 0.0;
    bad = 0;
  }
  for (int idx = tid; idx < NB * NB; idx += blockDim.x) {
    const int i = idx / NB, j = idx % NB;
    float v;
    if (i < b && j < b)
      v = (j <= i) ? W[(o + i) * ldw + (o + j)] : 0.f;
    else
      v = (i == j) ? 1.f : 0.f;
    s[i][j] = v;
  }
  __syncthreads();
  if (tid == 0 && fault == FFH_FAULT_BAD_PIVOT && p == 0) s[0][0] = __int_as_float(0x7fc00000);
  for (int j = 0; j < NB; ++j) {
    __syncthreads();
    if (tid == 0) {
      float dj = s[j][j];
      if (!(dj > 0.f) || !isfinite(dj)) {
        if (!bad) {
          bad = 1;
          raise_error(st, FFH_ERR_NOT_SPD, (int)(o + j));
        }
        dj = 1.f;
      }
      const float r = sqrtf(dj);
      s[j][j] = r;
      if (j < b) ld_acc += 2.0 * (double)logf(r);
    }
    __syncthreads();
    const float rinv = 1.f / s[j][j];
    for (int i = j + 1 + tid; i < NB; i += blockDim.x) s[i][j] *= rinv;
    __syncthreads();
    const int w = NB - 1 - j;
    for (int idx = tid; idx < w * w; idx += blockDim.x) {
      const int i = j + 1 + idx / w, k = j + 1 + idx % w;
      if (k <= i) s[i][k] = fmaf(-s[i][j], s[k][j], s[i][k]);
    }
  }
  __syncthreads();
  // inverse of the lower-triangular factor, one column per thread
  if (tid < NB) {
    const int c = tid;
    for (int i = 0; i < NB; ++i) {
      if (i < c) {
        inv[i][c] = 0.f;
        continue;
      }
      float acc = (i == c) ? 1.f : 0.f;
      for (int k = c; k < i; ++k) acc = fmaf(-s[i][k], inv[k][c], acc);
      inv[i][c] = acc / s[i][i];
    }
  }
  __syncthreads();
  for (int idx = tid; idx < NB * NB; idx += blockDim.x) {
    const int i = idx / NB, j = idx % NB;
    DI[idx] = inv[i][j];
    if (i < b && j < b) L[(o + i) * ldl + (o + j)] = (j <= i) ? s[i][j] : 0.f;
  }
  if (tid == 0) atomicAdd(&st->logdet, ld_acc);
}

__global__ void k_place_diag(const float* DI, int nt, int64_t d, float* M, int64_t ldm) {
  const int p = blockIdx.x;
  const int64_t o = (int64_t)p * NB;
  const int b = (int)((d - o) < NB ? (d - o) : NB);
  for (int idx = threadIdx.x; idx < NB * NB; idx += blockDim.x) {
    const int i = idx / NB, j = idx % NB;
    if (i < b && j < b) M[(o + i) * ldm + (o + j)] = DI[(int64_t)p * NB * NB + idx];
  }
}

size_t cholesky_work_floats(int64_t d) {
  // W (d x d copy of F) + T scratch for the inverse (<= d*d/2 + one block) + slack
  return (size_t)d * d + (size_t)d * d / 2 + (size_t)NB * NB * 4 + 1024;
}

cudaError_t launch_cholesky(const float* F, int64_t d, int64_t ldf, float* L, float* Linv,
                            float* work, float* DI, DevStatus* st, int fault, cudaStream_t s) {
  cudaError_t e;
  float* W = work;                 // d x d, pitch d
  float* Tmp = work + (size_t)d * d;
  e = cudaMemcpy2DAsync(W, d * sizeof(float), F, ldf * sizeof(float), d * sizeof(float), d,
                        cudaMemcpyDeviceToDevice, s);
  if (e != cudaSuccess) return e;
  e = cudaMemsetAsync(L, 0, (size_t)d * d * sizeof(float), s);
  if (e != cudaSuccess) return e;
  e = cudaMemsetAsync(&st->logdet, 0, sizeof(double), s);
  if (e != cudaSuccess) return e;
  const int nt = (int)((d + NB - 1) / NB);
  for (int p = 0; p < nt; ++p) {
    const int64_t o = (int64_t)p * NB;
    k_chol_diag<<<1, 256, 0, s>>>(W, d, d, p, L, d, DI + (size_t)p * NB * NB, st, fault); note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const int64_t rows = d - o - NB;
    if (rows <= 0) continue;
    // panel: L21 = W21 * L11^-T
    GemmArgs t{};
    t.A = W + (o + NB) * d + o;
    t.lda = d;
    t.B = DI + (size_t)p * NB * NB;
    t.ldb = NB;
    t.C = L + (o + NB) * d + o;
    t.ldc = d;
    t.M = (int)rows;
    t.N = NB;
    t.K = NB;
    t.alpha = 1.f;
    t.beta = 0.f;
    t.flags = GF_TRANS_B | GF_B_LOWER_NT;
    if ((e = gemm(t, 1, s)) != cudaSuccess) return e;
    // trailing update (lower tiles): W22 -= L21 L21^T
    GemmArgs u{};
    u.A = L + (o + NB) * d + o;
    u.lda = d;
    u.B = L + (o + NB) * d + o;
    u.ldb = d;
    u.C = W + (o + NB) * d + (o + NB);
    u.ldc = d;
    u.M = (int)rows;
    u.N = (int)rows;
    u.K = NB;
    u.alpha = -1.f;
    u.beta = 1.f;
    u.flags = GF_TRANS_B | GF_LOWER_C;
    if ((e = gemm(u, 1, s)) != cudaSuccess) return e;
  }
  if (!Linv) return cudaSuccess;
  // M = L^-1 by recursive doubling
  e = cudaMemsetAsync(Linv, 0, (size_t)d * d * sizeof(float), s);
  if (e != cudaSuccess) return e;
  k_place_diag<<<nt, 256, 0, s>>>(DI, nt, d, Linv, d); note_launches(1);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  for (int64_t b = NB; b < d; b *= 2) {
    const int64_t full_pairs = d / (2 * b);
    const int64_t o_last = full_pairs * 2 * b;
    const int64_t rows_last = d - o_last - b;  // rows of the trailing partial pair
    for (int part = 0; part < 2; ++part) {
      const int64_t batch = part == 0 ? full_pairs : (rows_last > 0 ? 1 : 0);
      if (batch == 0) continue;
      const int64_t o = part == 0 ? 0 : o_last;
      const int64_t rows = part == 0 ? b : rows_last;
      // Tmp_z = L21 * M11   (M11 lower: op(B)[k][c] = 0 for k < c)
      GemmArgs t{};
      t.A = L + (o + b) * d + o;
      t.lda = d;
      t.strideA = 2 * b * d + 2 * b;
      t.B = Linv + o * d + o;
      t.ldb = d;
      t.strideB = 2 * b * d + 2 * b;
      t.C = Tmp;
      t.ldc = b;
      t.strideC = b * b;
      t.M = (int)rows;
      t.N = (int)b;
      t.K = (int)b;
      t.alpha = 1.f;
      t.beta = 0.f;
      t.flags = GF_B_LOWER_NN;
      if ((e = gemm(t, (int)batch, s)) != cudaSuccess) return e;
      // M21 = -M22 * Tmp_z   (M22 lower)
      GemmArgs u{};
      u.A = Linv + (o + b) * d + (o + b);
      u.lda = d;
      u.strideA = 2 * b * d + 2 * b;
      u.B = Tmp;
      u.ldb = b;
      u.strideB = b * b;
      u.C = Linv + (o + b) * d + o;
      u.ldc = d;
      u.strideC = 2 * b * d + 2 * b;
      u.M = (int)rows;
      u.N = (int)b;
      u.K = (int)rows;
      u.alpha = -1.f;
      u.beta = 0.f;
      u.flags = GF_A_LOWER;
      if ((e = gemm(u, (int)batch, s)) != cudaSuccess) return e;
    }
  }
  return cudaSuccess;
}

// ---------------------------------------------------------------------------
// small kernels
// ---------------------------------------------------------------------------
__global__ void k_fill_identity(float* F, int64_t d, int64_t ld) {
  const int64_t total = d * d;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int64_t r = idx / d, c = idx - r * d;
    F[r * ld + c] = (r == c) ? 1.f : 0.f;
  }
}

cudaError_t launch_fill_identity(float* F, int64_t d, int64_t ld, cudaStream_t s) {
  const int64_t blocks = std::min<int64_t>((d * d + 255) / 256, (int64_t)num_sms() * 16);
  k_fill_identity<<<(unsigned)std::max<int64_t>(1, blocks), 256, 0, s>>>(F, d, ld); note_launches(1);
  return cudaGetLastError();
}

// F += lambda * mean(diag F) * I (mean taken before the shift); the shift is also
// written to *shift_out when given
__global__ void k_damp(float* F, int64_t d, int64_t ld, float lambda, double* shift_out) {
  double acc = 0.0;
  for (int64_t i = threadIdx.x; i < d; i += blockDim.x) acc += F[i * ld + i];
  __shared__ double tot;
  const double sum = block_sum_f64(acc);
  if (threadIdx.x == 0) tot = sum;
  __syncthreads();
  const float shift = (float)((double)lambda * tot / (double)d);
  for (int64_t i = threadIdx.x; i < d; i += blockDim.x) F[i * ld + i] += shift;
  if (threadIdx.x == 0 && shift_out) *shift_out = (double)shift;
}

cudaError_t launch_damp(float* F, int64_t d, int64_t ld, float lambda, DevStatus*,
                        cudaStream_t s, double* shift_out) {
  if (lambda == 0.f) return shift_out ? cudaMemsetAsync(shift_out, 0, sizeof(double), s)
                                      : cudaSuccess;
  k_damp<<<1, 1024, 0, s>>>(F, d, ld, lambda, shift_out);
  note_launches(1);
  return cudaGetLastError();
}

// C += X (d x d, same pitch)
__global__ void k_add(float* C, const float* X, int64_t total) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x)
    C[i] += X[i];
}

cudaError_t launch_add(float* C, const float* X, int64_t total, cudaStream_t s) {
  const int64_t blocks = std::min<int64_t>((total + 255) / 256, (int64_t)num_sms() * 8);
  k_add<<<(unsigned)std::max<int64_t>(1, blocks), 256, 0, s>>>(C, X, total);
  note_launches(1);
  return cudaGetLastError();
}

// s = tr(A)/n, trB; stored into the record
__global__ void k_norm_trace(const float* A, int64_t n, const float* B, int64_t m,
                             IterRecord* rec) {
  double a = 0.0, b = 0.0;
  for (int64_t i = threadIdx.x; i < n; i += blockDim.x) a += A[i * n + i];
  for (int64_t i = threadIdx.x; i < m; i += blockDim.x) b += B[i * m + i];
  const double sa = block_sum_f64(a);
  __syncthreads();
  const double sb = block_sum_f64(b);
  if (threadIdx.x == 0) {
    const double sc = sa / (double)n;
    rec->scale = sc;
    rec->trB = sb * sc;
  }
}

__global__ void k_norm_apply(float* A, int64_t n, float* B, int64_t m, const IterRecord* rec) {
  const double sc = rec->scale;
  const float ia = (float)(1.0 / sc), sb = (float)sc;
  const int64_t tot_a = n * n, tot_b = m * m;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < tot_a + tot_b;
       idx += (int64_t)gridDim.x * blockDim.x) {
    if (idx < tot_a)
      A[idx] *= ia;
    else
      B[idx - tot_a] *= sb;
  }
}

cudaError_t launch_normalize(float* A, int64_t n, float* B, int64_t m, IterRecord* rec,
                             DevStatus*, cudaStream_t s) {
  k_norm_trace<<<1, 1024, 0, s>>>(A, n, B, m, rec); note_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t tot = n * n + m * m;
  const int64_t blocks = std::min<int64_t>((tot + 255) / 256, (int64_t)num_sms() * 16);
  k_norm_apply<<<(unsigned)blocks, 256, 0, s>>>(A, n, B, m, rec); note_launches(1);
  return cudaGetLastError();
}

// sum (F/trF - P/trP)^2 and sum (F/trF)^2 (trF, trP read from device doubles).  Per
// element in fp32, float4 loads, per-thread partial sums (a few dozen terms) in fp32 and
// the block and grid sums in fp64: FP64 arithmetic per element is slow on this part, and
// the statistic needs only a few significant digits.
__global__ void k_delta(const float* F, const float* P, int64_t total, const double* trF,
                        const double* trP, double* d2, double* n2) {
  const float a = (float)(1.0 / *trF), b = (float)(1.0 / *trP);
  float sdf = 0.f, snf = 0.f;
  const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const bool vec = ((reinterpret_cast<uintptr_t>(F) | reinterpret_cast<uintptr_t>(P)) & 15) == 0;
  const int64_t n4 = vec ? total / 4 : 0;
  for (int64_t i = t0; i < n4; i += stride) {
    const float4 fv = reinterpret_cast<const float4*>(F)[i];
    const float4 pv = reinterpret_cast<const float4*>(P)[i];
    const float f[4] = {fv.x * a, fv.y * a, fv.z * a, fv.w * a};
    const float p[4] = {pv.x * b, pv.y * b, pv.z * b, pv.w * b};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float dd = f[e] - p[e];
      sdf = fmaf(dd, dd, sdf);
      snf = fmaf(f[e], f[e], snf);
    }
  }
  for (int64_t idx = 4 * n4 + t0; idx < total; idx += stride) {
    const float f = F[idx] * a, p = P[idx] * b;
    sdf = fmaf(f - p, f - p, sdf);
    snf = fmaf(f, f, snf);
  }
  double sd = block_sum_f64((double)sdf), sn;
  __syncthreads();
  sn = block_sum_f64((double)snf);
  if (threadIdx.x == 0) {
    atomicAdd(d2, sd);
    atomicAdd(n2, sn);
  }
}

cudaError_t launch_delta(const float* F, const float* Fprev, int64_t d, double* d2, double* n2,
                         double* tr, cudaStream_t s) {
  // tr[0] = tr(F), tr[1] = tr(Fprev)
  const int64_t tot = d * d;
  const int64_t blocks = std::min<int64_t>((tot + 255) / 256, (int64_t)num_sms() * 8);
  k_delta<<<(unsigned)std::max<int64_t>(1, blocks), 256, 0, s>>>(F, Fprev, tot, tr, tr + 1, d2,
                                                                  n2); note_launches(1);
  return cudaGetLastError();
}

__global__ void k_trace_f64(const float* F, int64_t d, double* out) {
  double a = 0.0;
  for (int64_t i = threadIdx.x; i < d; i += blockDim.x) a += F[i * d + i];
  a = block_sum_f64(a);
  if (threadIdx.x == 0) *out = a;
}

cudaError_t launch_trace(const float* F, int64_t d, double* out, cudaStream_t s) {
  k_trace_f64<<<1, 1024, 0, s>>>(F, d, out); note_launches(1);
  return cudaGetLastError();
}

__global__ void k_dot(const float* a, const float* b, int64_t N, double* out) {
  double acc = 0.0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < N;
       i += (int64_t)gridDim.x * blockDim.x)
    acc += (double)a[i] * (double)b[i];
  acc = block_sum_f64(acc);
  if (threadIdx.x == 0) atomicAdd(out, acc);
}

cudaError_t launch_dot(const float* a, const float* b, int64_t N, double* out, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(out, 0, sizeof(double), s);
  if (e != cudaSuccess) return e;
  const int64_t blocks = std::min<int64_t>((N + 255) / 256, (int64_t)num_sms() * 4);
  k_dot<<<(unsigned)std::max<int64_t>(1, blocks), 256, 0, s>>>(a, b, N, out); note_launches(1);
  return cudaGetLastError();
}

// ||F||_F^2
__global__ void k_frob2(const float* F, int64_t total, double* out) {
  double acc = 0.0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x)
    acc += (double)F[i] * (double)F[i];
  acc = block_sum_f64(acc);
  if (threadIdx.x == 0) atomicAdd(out, acc);
}

cudaError_t launch_frob2(const float* F, int64_t d, double* out, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(out, 0, sizeof(double), s);
  if (e != cudaSuccess) return e;
  const int64_t tot = d * d;
  const int64_t blocks = std::min<int64_t>((tot + 255) / 256, (int64_t)num_sms() * 4);
  k_frob2<<<(unsigned)std::max<int64_t>(1, blocks), 256, 0, s>>>(F, tot, out); note_launches(1);
  return cudaGetLastError();
}

// F *= 1 / *denom
__global__ void k_scale_by_inv(float* F, int64_t total, const double* denom) {
  const float f = (float)(1.0 / *denom);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x)
    F[i] *= f;
}

cudaError_t launch_scale_by_inv(float* F, int64_t d, const double* denom, cudaStream_t s) {
  const int64_t tot = d * d;
  const int64_t blocks = std::min<int64_t>((tot + 255) / 256, (int64_t)num_sms() * 16);
  k_scale_by_inv<<<(unsigned)std::max<int64_t>(1, blocks), 256, 0, s>>>(F, tot, denom); note_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// CUDA-core weighted Gram and quadratic forms (cross-check path, option kernel=1)
// ---------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) k_gram_simt(const T* __restrict__ V, int64_t N, int64_t d,
                                                   int64_t ld, const float* __restrict__ w,
                                                   float scale, float* C, int64_t ldc) {
  const int row0 = blockIdx.y * 64, col0 = blockIdx.x * 64;
  if (col0 > row0 + 63) return;
  __shared__ float As[16][68];
  __shared__ float Bs[16][68];
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  float acc[4][4] = {};
  for (int64_t k0 = 0; k0 < N; k0 += 16) {
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int idx = tid + e * 256;
      const int kk = idx >> 6, c = idx & 63;
      const int64_t k = k0 + kk;
      float a = 0.f, b = 0.f;
      if (k < N) {
        const float wk = w ? w[k] : 1.f;
        if (row0 + c < d) a = ldf(V + k * ld + row0 + c) * wk;
        if (col0 + c < d) b = ldf(V + k * ld + col0 + c);
      }
      As[kk][c] = a;
      Bs[kk][c] = b;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t r = row0 + ty * 4 + i;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t c = col0 + tx * 4 + j;
      if (r < d && c < d && c <= r) {
        const float v = acc[i][j] * scale;
        C[r * ldc + c] = v;
        C[c * ldc + r] = v;
      }
    }
  }
}

cudaError_t launch_gram_simt(const void* V, int dtype, int64_t N, int64_t d, int64_t ld,
                             const float* w, float scale, float* C, int64_t ldc, cudaStream_t s) {
  const int nt = (int)((d + 63) / 64);
  dim3 grid(nt, nt);
  if (dtype == FFH_BF16) {
    k_gram_simt<<<grid, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(V), N, d, ld, w, scale, C,
                                     ldc);
  } else {
    k_gram_simt<<<grid, 256, 0, s>>>(static_cast<const float*>(V), N, d, ld, w, scale, C, ldc);
  }
  note_launches(1);
  return cudaGetLastError();
}

// q_k = ||M v_k||^2 (M lower, fp32) or, with FWD, v_k^T F v_k (F full, fp32).
// One CTA per 64 samples; loops over 64-wide output chunks.
template <typename T, bool FWD>
__global__ void __launch_bounds__(256) k_qform_simt(const T* __restrict__ V, int64_t N,
                                                    int64_t d, int64_t ld,
                                                    const float* __restrict__ M, int64_t ldm,
                                                    float* __restrict__ q) {
  const int64_t row0 = (int64_t)blockIdx.x * 64;
  __shared__ float As[16][68];
  __shared__ float Bs[16][68];
  __shared__ float rowacc[64][17];
  const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
  float part[4] = {0.f, 0.f, 0.f, 0.f};
  for (int64_t c0 = 0; c0 < d; c0 += 64) {
    float acc[4][4] = {};
    const int64_t khi = FWD ? d : ((c0 + 64) < d ? (c0 + 64) : d);
    for (int64_t k0 = 0; k0 < khi; k0 += 16) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int idx = tid + e * 256;
        const int r = idx >> 4, kk = idx & 15;
        const int64_t gr = row0 + r, gk = k0 + kk;
        As[kk][r] = (gr < N && gk < khi) ? ldf(V + gr * ld + gk) : 0.f;
        const int c = idx >> 4;  // output index within the chunk
        const int64_t gc = c0 + c;
        Bs[kk][c] = (gc < d && gk < khi) ? M[gc * ldm + gk] : 0.f;
      }
      __syncthreads();
#pragma unroll
      for (int kk = 0; kk < 16; ++kk) {
        float a[4], b[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
        for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
      }
      __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int64_t gc = c0 + tx * 4 + j;
        if (gc >= d) continue;
        if (FWD) {
          const int64_t gr = row0 + ty * 4 + i;
          const float x = gr < N ? ldf(V + gr * ld + gc) : 0.f;
          part[i] = fmaf(acc[i][j], x, part[i]);
        } else {
          part[i] = fmaf(acc[i][j], acc[i][j], part[i]);
        }
      }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) rowacc[ty * 4 + i][tx] = part[i];
  __syncthreads();
  if (tid < 64) {
    float s = 0.f;
    for (int j = 0; j < 16; ++j) s += rowacc[tid][j];
    const int64_t gr = row0 + tid;
    if (gr < N) q[gr] = s;
  }
}

cudaError_t launch_qform_simt(const void* V, int dtype, int64_t N, int64_t d, int64_t ld,
                              const float* M, int64_t ldm, float* q, cudaStream_t s) {
  const int64_t blocks = (N + 63) / 64;
  if (blocks == 0) return cudaSuccess;
  if (dtype == FFH_BF16) {
    k_qform_simt<__nv_bfloat16, false><<<(unsigned)blocks, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(V), N, d, ld, M, ldm, q);
  } else {
    k_qform_simt<float, false>
        <<<(unsigned)blocks, 256, 0, s>>>(static_cast<const float*>(V), N, d, ld, M, ldm, q);
  }
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_fwd_qform_simt(const void* V, int dtype, int64_t N, int64_t d, int64_t ld,
                                  const float* F, int64_t ldf, float* q, cudaStream_t s) {
  const int64_t blocks = (N + 63) / 64;
  if (blocks == 0) return cudaSuccess;
  if (dtype == FFH_BF16) {
    k_qform_simt<__nv_bfloat16, true><<<(unsigned)blocks, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(V), N, d, ld, F, ldf, q);
  } else {
    k_qform_simt<float, true>
        <<<(unsigned)blocks, 256, 0, s>>>(static_cast<const float*>(V), N, d, ld, F, ldf, q);
  }
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_zero_f64(double* p, int n, cudaStream_t s) {
  return cudaMemsetAsync(p, 0, sizeof(double) * n, s);
}

}  // namespace ffh
