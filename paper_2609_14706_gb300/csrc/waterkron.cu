// WaterKron downstream of the fit (Sections 2 and 3): reverse Cholesky, waterfilling
// scales (Corollary 3.2) and the two-sided GPTQ quantizer (Algorithm 2).
//
// Reverse Cholesky (Section 2 notation, L lower with L^T L = F): with the reversal J,
//   C C^T = J F J (ordinary Cholesky, the tensor-core factorization of this library) gives
//   L = J C^T J, and L^-1 = J C^-T J from C^-1, column-normalised for Algorithms 1-2.
//
// Two-sided GPTQ: columns j = 0..n-1, rows i = 0..m-1 in turn,
//   Z_ij = round(W_ij / (alpha_j beta_i)),  Delta_ij = alpha_j beta_i Z_ij - W_ij,
//   W <- W + Lt^B[:, i] Delta_ij Lt^A[:, j]^T.
// With Lt lower unit-triangular, entry (i, j) sees the feedback of every (i', j') with
// i' <= i and j' <= j, which splits into
//   * the earlier columns j' < j: sum_j' u_j'[i] Lt^A[j][j'], with u_j' = Lt^B Delta_{:,j'}
//     the total change of column j' (final for row i once column j' has passed row i);
//   * the earlier rows of column j: sum_{i' < i} Lt^B[i][i'] Delta_i'j.
// So columns can run as a wavefront: column j processes 32-row blocks in order, each one
// after column j-1 has finished the same block.  Columns go in blocks of 128 (one CTA per
// column, k_gptq2_block); the earlier column blocks' feedback is applied between blocks by
// an fp32 GEMM (k_gemm_nt_f32).
#include <algorithm>

#include "ffh_internal.cuh"

namespace ffh {

static constexpr uint64_t kFlagWaitNs = 4000000000ull;  // bounded wait on a peer CTA
constexpr int kQBlockCols = 128;                       // columns per wavefront launch

__device__ __forceinline__ uint64_t wk_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ int ld_acquire(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(int* p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// ---------------------------------------------------------------------------
// out[i][j] = F[d-1-i][d-1-j]  (J F J), row-major, pitch d
// ---------------------------------------------------------------------------
__global__ void k_reverse_sym(const float* __restrict__ F, int64_t d, int64_t ldf,
                              float* __restrict__ out) {
  const int64_t total = d * d;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = idx / d, j = idx - i * d;
    out[idx] = F[(d - 1 - i) * ldf + (d - 1 - j)];
  }
}

// out[i][j] = C[d-1-j][d-1-i] (lower part, zeros above), optionally divided by
// C[d-1-j][d-1-j] (the diagonal of out's column j).  32 x 32 tiles through shared memory.
__global__ void k_rev_transpose(const float* __restrict__ C, int64_t d, float* __restrict__ out,
                                int normalize) {
  __shared__ float tile[32][33];
  const int64_t ti = blockIdx.y, tj = blockIdx.x;
  if (tj > ti) {
    // strictly above the diagonal: zeros
    for (int y = threadIdx.y; y < 32; y += 8) {
      const int64_t i = ti * 32 + y, j = tj * 32 + threadIdx.x;
      if (i < d && j < d) out[i * d + j] = 0.f;
    }
    return;
  }
  // out rows i = 32 ti + x, cols j = 32 tj + y  <-  C[d-1-j][d-1-i]
  for (int y = threadIdx.y; y < 32; y += 8) {
    const int64_t i = ti * 32 + threadIdx.x, j = tj * 32 + y;
    tile[y][threadIdx.x] = (i < d && j < d) ? C[(d - 1 - j) * d + (d - 1 - i)] : 0.f;
  }
  __syncthreads();
  for (int y = threadIdx.y; y < 32; y += 8) {
    const int64_t i = ti * 32 + y, j = tj * 32 + threadIdx.x;
    if (i < d && j < d) {
      float v = (j <= i) ? tile[threadIdx.x][y] : 0.f;
      if (normalize && j <= i) v /= C[(d - 1 - j) * d + (d - 1 - j)];
      out[i * d + j] = v;
    }
  }
}

cudaError_t launch_rev_transpose(const float* C, int64_t d, float* out, bool normalize,
                                 cudaStream_t s) {
  const unsigned nt = (unsigned)((d + 31) / 32);
  k_rev_transpose<<<dim3(nt, nt), dim3(32, 8), 0, s>>>(C, d, out, normalize ? 1 : 0);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_reverse_sym(const float* F, int64_t d, int64_t ldf, float* out,
                               cudaStream_t s) {
  const int64_t blocks = std::min<int64_t>((d * d + 255) / 256, (int64_t)num_sms() * 16);
  k_reverse_sym<<<(unsigned)std::max<int64_t>(1, blocks), 256, 0, s>>>(F, d, ldf, out);
  note_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Corollary 3.2: alpha_j = sqrt(gamma) |A|^(1/2n) / L^A_jj, |A|^(1/2n) = geometric mean of
// diag(L^A); the same for beta with L^B.  One block per factor.
// ---------------------------------------------------------------------------
__global__ void k_waterfilling(const float* LA, int64_t n, const float* LB, int64_t m, float gamma,
                               float* alpha, float* beta) {
  const float* L = blockIdx.x == 0 ? LA : LB;
  const int64_t d = blockIdx.x == 0 ? n : m;
  float* out = blockIdx.x == 0 ? alpha : beta;
  __shared__ double red[32];
  double s = 0.0;
  for (int64_t i = threadIdx.x; i < d; i += blockDim.x) s += (double)logf(L[i * d + i]);
  for (int o = 16; o > 0; o >>= 1) s += __shfl_down_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x < 32) {
    s = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0;
    for (int o = 16; o > 0; o >>= 1) s += __shfl_down_sync(0xffffffffu, s, o);
    if (threadIdx.x == 0) red[0] = s;
  }
  __syncthreads();
  const float g = (float)exp(red[0] / (double)d) * sqrtf(gamma);
  for (int64_t i = threadIdx.x; i < d; i += blockDim.x) out[i] = g / L[i * d + i];
}

cudaError_t launch_waterfilling(const float* LA, int64_t n, const float* LB, int64_t m,
                                float gamma, float* alpha, float* beta, cudaStream_t s) {
  k_waterfilling<<<2, 1024, 0, s>>>(LA, n, LB, m, gamma, alpha, beta);
  note_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// two-sided GPTQ: one column block of up to kQBlockCols columns, one CTA per column
// ---------------------------------------------------------------------------
struct Gptq2Args {
  float* W;            // m x n working copy (pitch n): earlier column blocks' feedback applied
  const float* LtA;    // n x n, column-normalised (RevCholesky(A))^-1, row-major
  const float* LtB;    // m x m, likewise for B
  const float* alpha;  // n
  const float* beta;   // m
  int32_t* Z;          // m x n
  float* V;            // m x n (optional): alpha_j beta_i Z_ij
  float* U;            // m x kQBlockCols: u_j = total change of column j (pitch kQBlockCols)
  int* flags;          // kQBlockCols x NI, zeroed: column c has finished row block I
  int64_t m, n;
  int J;               // first column of the block
  int NI;              // 32-row blocks
  DevStatus* st;
};

__global__ void __launch_bounds__(256) k_gptq2_block(const Gptq2Args a) {
  extern __shared__ float delta[];  // [m]: Delta_ij of this column, rows processed so far
  __shared__ float wb[32], w0b[32];
  __shared__ int stop;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c = blockIdx.x;
  const int64_t j = a.J + c, m = a.m, n = a.n;
  const float aj = a.alpha[j];
  if (tid == 0) stop = 0;
  __syncthreads();
  for (int I = 0; I < a.NI; ++I) {
    const int64_t r0 = (int64_t)I * 32;
    const int rb = (int)((m - r0) < 32 ? (m - r0) : 32);
    // the previous column of the block has finished this row block (bounded wait)
    if (c > 0 && tid == 0) {
      const int* f = a.flags + (int64_t)(c - 1) * a.NI + I;
      if (ld_acquire(f) == 0) {
        const uint64_t t0 = wk_timer_ns();
        while (ld_acquire(f) == 0) {
          if (*reinterpret_cast<volatile int*>(&a.st->abort_all)) {
            stop = 1;
            break;
          }
          if (wk_timer_ns() - t0 > kFlagWaitNs) {
            raise_error(a.st, FFH_ERR_TIMEOUT, 31);
            stop = 1;
            break;
          }
          __nanosleep(200);
        }
      }
    }
    __syncthreads();
    if (stop) break;
    // feedback into rows r0..r0+rb-1 of column j: one warp per row, contiguous float4
    // reads of the row of Lt^B
    for (int kk = warp; kk < rb; kk += 8) {
      const int64_t r = r0 + kk;
      float sc = 0.f, sw = 0.f;
      // earlier columns of this block: sum_c' u_{J+c'}[r] Lt^A[j][J+c']
      for (int cc = lane; cc < c; cc += 32)
        sc = fmaf(a.U[r * kQBlockCols + cc], a.LtA[j * n + a.J + cc], sc);
      // earlier rows of this column: sum_{i < r0} Lt^B[r][i] Delta_i
      const float* lrow = a.LtB + r * m;
      if ((m & 3) == 0) {
        for (int64_t i = 4 * lane; i < r0; i += 128) {
          const float4 lv = *reinterpret_cast<const float4*>(lrow + i);
          const float4 dv = *reinterpret_cast<const float4*>(delta + i);
          sw = fmaf(lv.x, dv.x, sw);
          sw = fmaf(lv.y, dv.y, sw);
          sw = fmaf(lv.z, dv.z, sw);
          sw = fmaf(lv.w, dv.w, sw);
        }
      } else {
        for (int64_t i = lane; i < r0; i += 32) sw = fmaf(lrow[i], delta[i], sw);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        sc += __shfl_xor_sync(0xffffffffu, sc, o);
        sw += __shfl_xor_sync(0xffffffffu, sw, o);
      }
      if (lane == 0) {
        const float w0 = a.W[r * n + j] + sc;
        w0b[kk] = w0;
        wb[kk] = w0 + sw;
      }
    }
    __syncthreads();
    if (warp == 0) {
      // the 32 rows of the block in turn (lane = row), Lt^B's diagonal block in registers
      const int64_t r = r0 + lane;
      const bool live = lane < rb;
      float w = live ? wb[lane] : 0.f;
      const float bl = live ? a.beta[r] : 1.f;
      float lt[32];
#pragma unroll
      for (int ii = 0; ii < 32; ++ii) lt[ii] = (live && ii < lane) ? a.LtB[r * m + r0 + ii] : 0.f;
      float z_my = 0.f, d_my = 0.f;
#pragma unroll
      for (int ii = 0; ii < 32; ++ii) {
        if (ii < rb) {
          const float wi = __shfl_sync(0xffffffffu, w, ii);
          const float s = aj * __shfl_sync(0xffffffffu, bl, ii);
          const float zi = rintf(wi / s);  // round to nearest, ties to even
          const float di = s * zi - wi;
          if (lane == ii) {
            z_my = zi;
            d_my = di;
            w = s * zi;  // W_ij + Delta = V_ij
          } else if (lane > ii) {
            w = fmaf(lt[ii], di, w);
          }
        }
      }
      if (live) {
        a.Z[r * n + j] = (int32_t)z_my;
        if (a.V) a.V[r * n + j] = w;
        delta[r] = d_my;
        a.U[r * kQBlockCols + c] = w - w0b[lane];
      }
    }
    __syncthreads();
    if (tid == 0) {
      __threadfence();
      st_release(a.flags + (int64_t)c * a.NI + I, 1);
    }
  }
}

// C[r][l] += sum_k A[r][k] B[l][k]: A = U (rows x K, pitch lda), B rows of Lt^A (pitch ldb),
// C = the remaining columns of W (pitch ldc).  64 x 64 tiles, 4 x 4 per thread.
__global__ void __launch_bounds__(256) k_gemm_nt_f32(const float* __restrict__ A, int64_t lda,
                                                     const float* __restrict__ B, int64_t ldb,
                                                     float* __restrict__ C, int64_t ldc,
                                                     int64_t rows, int64_t cols, int K) {
  __shared__ float As[64][65], Bs[64][65];
  const int64_t r0 = (int64_t)blockIdx.y * 64, c0 = (int64_t)blockIdx.x * 64;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 64) {
    for (int e = threadIdx.x; e < 64 * 64; e += 256) {
      const int rr = e >> 6, kk = e & 63;
      As[rr][kk] = (r0 + rr < rows && k0 + kk < K) ? A[(r0 + rr) * lda + k0 + kk] : 0.f;
      Bs[rr][kk] = (c0 + rr < cols && k0 + kk < K) ? B[(c0 + rr) * ldb + k0 + kk] : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < 64; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[ty * 4 + i][kk];
#pragma unroll
      for (int jx = 0; jx < 4; ++jx) bv[jx] = Bs[tx * 4 + jx][kk];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int jx = 0; jx < 4; ++jx) acc[i][jx] = fmaf(av[i], bv[jx], acc[i][jx]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int jx = 0; jx < 4; ++jx) {
      const int64_t r = r0 + ty * 4 + i, cc = c0 + tx * 4 + jx;
      if (r < rows && cc < cols) C[r * ldc + cc] += acc[i][jx];
    }
}

size_t gptq2_work_bytes(int64_t m, int64_t n) {
  const int64_t NI = (m + 31) / 32;
  return (size_t)m * n * 4 + (size_t)m * kQBlockCols * 4 + (size_t)kQBlockCols * NI * 4 + 1024;
}

cudaError_t launch_gptq2(const float* W, const float* LtA, const float* LtB, const float* alpha,
                         const float* beta, int64_t m, int64_t n, int32_t* Z, float* V,
                         void* work, DevStatus* st, cudaStream_t s) {
  cudaError_t e;
  const int NI = (int)((m + 31) / 32);
  char* wp = static_cast<char*>(work);
  float* Wk = reinterpret_cast<float*>(wp);
  wp += (size_t)m * n * 4;
  float* U = reinterpret_cast<float*>(wp);
  wp += (size_t)m * kQBlockCols * 4;
  int* flags = reinterpret_cast<int*>(wp);
  const size_t smem = (size_t)m * 4;
  if (smem > 48 * 1024 &&
      (e = cudaFuncSetAttribute(k_gptq2_block, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)smem)) != cudaSuccess)
    return e;
  if ((e = cudaMemcpyAsync(Wk, W, (size_t)m * n * 4, cudaMemcpyDeviceToDevice, s)) != cudaSuccess)
    return e;
  for (int64_t J = 0; J < n; J += kQBlockCols) {
    const int ncol = (int)std::min<int64_t>(kQBlockCols, n - J);
    if ((e = cudaMemsetAsync(flags, 0, sizeof(int) * kQBlockCols * NI, s)) != cudaSuccess) return e;
    Gptq2Args a;
    a.W = Wk;
    a.LtA = LtA;
    a.LtB = LtB;
    a.alpha = alpha;
    a.beta = beta;
    a.Z = Z;
    a.V = V;
    a.U = U;
    a.flags = flags;
    a.m = m;
    a.n = n;
    a.J = (int)J;
    a.NI = NI;
    a.st = st;
    k_gptq2_block<<<ncol, 256, smem, s>>>(a);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const int64_t rest = n - J - ncol;
    if (rest > 0) {
      // W[:, J+ncol:] += U[:, :ncol] Lt^A[J+ncol:, J:J+ncol]^T
      k_gemm_nt_f32<<<dim3((unsigned)((rest + 63) / 64), (unsigned)((m + 63) / 64)), 256, 0, s>>>(
          U, kQBlockCols, LtA + (J + ncol) * n + J, n, Wk + J + ncol, n, m, rest, ncol);
      note_launches(1);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
  }
  return cudaSuccess;
}

}  // namespace ffh
