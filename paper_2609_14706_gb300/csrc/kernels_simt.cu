// Small CUDA-core kernels of the FlipFlop Hessian fit: conversions, the A_0 = I
// shortcut q_k = ||x_k||^2, damping, trace normalisation, the convergence statistics
// and fp64 dot products.  The N-sized passes and the Cholesky run on the tensor cores
// (kernels_tc.cu, kernels_chol.cu).
#include <algorithm>
#include <atomic>

#include "ffh_internal.cuh"

namespace ffh {

static std::atomic<long long> g_launches{0};
void note_launches(int k) { g_launches.fetch_add(k, std::memory_order_relaxed); }
long long launches_so_far() { return g_launches.load(std::memory_order_relaxed); }

static thread_local const DevStatus* t_gate = nullptr;
const DevStatus* current_gate() { return t_gate; }
void set_current_gate(const DevStatus* st) { t_gate = st; }

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
                          __nv_bfloat16* __restrict__ dst, int64_t ldd, int lower,
                          const DevStatus* gate) {
  if (gated_off(gate)) return;
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
  k_to_bf16<<<(unsigned)blocks, 256, 0, s>>>(src, rows, cols, lds, dst, ldd, lower,
                                               current_gate());
  note_launches(1);
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
                                 __nv_bfloat16* __restrict__ dst, int64_t ldd,
                                 const DevStatus* gate) {
  if (gated_off(gate)) return;
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
  k_lowerT_to_bf16<<<dim3(nb, nb), dim3(32, 8), 0, s>>>(src, d, lds, dst, ldd, current_gate());
  note_launches(1);
  return cudaGetLastError();
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
__global__ void k_damp(float* F, int64_t d, int64_t ld, float lambda, double* shift_out,
                       const DevStatus* gate) {
  if (gated_off(gate)) return;
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
  k_damp<<<1, 1024, 0, s>>>(F, d, ld, lambda, shift_out, current_gate());
  note_launches(1);
  return cudaGetLastError();
}

// C += X (d x d, same pitch)
__global__ void k_add(float* C, const float* X, int64_t total, const DevStatus* gate) {
  if (gated_off(gate)) return;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x)
    C[i] += X[i];
}

cudaError_t launch_add(float* C, const float* X, int64_t total, cudaStream_t s) {
  const int64_t blocks = std::min<int64_t>((total + 255) / 256, (int64_t)num_sms() * 8);
  k_add<<<(unsigned)std::max<int64_t>(1, blocks), 256, 0, s>>>(C, X, total, current_gate());
  note_launches(1);
  return cudaGetLastError();
}

// s = tr(A)/n, trB; stored into the record
__global__ void k_norm_trace(const float* A, int64_t n, const float* B, int64_t m,
                             IterRecord* rec, const DevStatus* gate) {
  if (gated_off(gate)) return;
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

__global__ void k_norm_apply(float* A, int64_t n, float* B, int64_t m, const IterRecord* rec,
                             const DevStatus* gate) {
  if (gated_off(gate)) return;
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
  k_norm_trace<<<1, 1024, 0, s>>>(A, n, B, m, rec, current_gate()); note_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t tot = n * n + m * m;
  const int64_t blocks = std::min<int64_t>((tot + 255) / 256, (int64_t)num_sms() * 16);
  k_norm_apply<<<(unsigned)blocks, 256, 0, s>>>(A, n, B, m, rec, current_gate());
  note_launches(1);
  return cudaGetLastError();
}

// sum (F/trF - P/trP)^2 and sum (F/trF)^2 (trF, trP read from device doubles).  Per
// element in fp32, float4 loads, per-thread partial sums (a few dozen terms) in fp32 and
// the block and grid sums in fp64: FP64 arithmetic per element is slow on this part, and
// the statistic needs only a few significant digits.
__global__ void k_delta(const float* F, const float* P, int64_t total, const double* trF,
                        const double* trP, double* red, const DevStatus* gate) {
  if (gated_off(gate)) return;
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
    red[2 * blockIdx.x] = sd;
    red[2 * blockIdx.x + 1] = sn;
  }
}

// out0 = sum_i red[nv i], out1 = sum_i red[nv i + 1] (nv = 1 or 2) over i < nb, in a fixed
// order (one block: thread t adds partials t, t + 256, ... in turn, then a fixed tree), so
// the fp64 statistics are the same on every run
__global__ void k_sum_partials(const double* red, int nb, int nv, double* out0, double* out1,
                               const DevStatus* gate) {
  if (gated_off(gate)) return;
  double a = 0.0, b = 0.0;
  for (int i = threadIdx.x; i < nb; i += blockDim.x) {
    a += red[(size_t)nv * i];
    if (nv == 2) b += red[(size_t)nv * i + 1];
  }
  a = block_sum_f64(a);
  __syncthreads();
  b = block_sum_f64(b);
  if (threadIdx.x == 0) {
    *out0 = a;
    if (out1) *out1 = b;
  }
}

static cudaError_t sum_partials(const double* red, int nb, int nv, double* out0, double* out1,
                                cudaStream_t s) {
  k_sum_partials<<<1, 256, 0, s>>>(red, nb, nv, out0, out1, current_gate());
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_delta(const float* F, const float* Fprev, int64_t d, double* d2, double* n2,
                         double* tr, double* red, cudaStream_t s) {
  // tr[0] = tr(F), tr[1] = tr(Fprev)
  const int64_t tot = d * d;
  const int64_t blocks = std::max<int64_t>(
      1, std::min<int64_t>({(tot + 255) / 256, (int64_t)num_sms() * 8, kRedDoubles / 2}));
  k_delta<<<(unsigned)blocks, 256, 0, s>>>(F, Fprev, tot, tr, tr + 1, red, current_gate());
  note_launches(1);
  cudaError_t e = cudaGetLastError();
  return e != cudaSuccess ? e : sum_partials(red, (int)blocks, 2, d2, n2, s);
}

__global__ void k_trace_f64(const float* F, int64_t d, double* out, const DevStatus* gate) {
  if (gated_off(gate)) return;
  double a = 0.0;
  for (int64_t i = threadIdx.x; i < d; i += blockDim.x) a += F[i * d + i];
  a = block_sum_f64(a);
  if (threadIdx.x == 0) *out = a;
}

cudaError_t launch_trace(const float* F, int64_t d, double* out, cudaStream_t s) {
  k_trace_f64<<<1, 1024, 0, s>>>(F, d, out, current_gate()); note_launches(1);
  return cudaGetLastError();
}

__global__ void k_dot(const float* a, const float* b, int64_t N, double* red,
                      const DevStatus* gate) {
  if (gated_off(gate)) return;
  double acc = 0.0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < N;
       i += (int64_t)gridDim.x * blockDim.x)
    acc += (double)a[i] * (double)b[i];
  acc = block_sum_f64(acc);
  if (threadIdx.x == 0) red[blockIdx.x] = acc;
}

cudaError_t launch_dot(const float* a, const float* b, int64_t N, double* out, double* red,
                       cudaStream_t s) {
  const int64_t blocks = std::max<int64_t>(
      1, std::min<int64_t>({(N + 255) / 256, (int64_t)num_sms() * 4, kRedDoubles}));
  k_dot<<<(unsigned)blocks, 256, 0, s>>>(a, b, N, red, current_gate());
  note_launches(1);
  cudaError_t e = cudaGetLastError();
  return e != cudaSuccess ? e : sum_partials(red, (int)blocks, 1, out, nullptr, s);
}

// ||F||_F^2
__global__ void k_frob2(const float* F, int64_t total, double* red, const DevStatus* gate) {
  if (gated_off(gate)) return;
  double acc = 0.0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x)
    acc += (double)F[i] * (double)F[i];
  acc = block_sum_f64(acc);
  if (threadIdx.x == 0) red[blockIdx.x] = acc;
}

cudaError_t launch_frob2(const float* F, int64_t d, double* out, double* red, cudaStream_t s) {
  const int64_t tot = d * d;
  const int64_t blocks = std::max<int64_t>(
      1, std::min<int64_t>({(tot + 255) / 256, (int64_t)num_sms() * 4, kRedDoubles}));
  k_frob2<<<(unsigned)blocks, 256, 0, s>>>(F, tot, red, current_gate());
  note_launches(1);
  cudaError_t e = cudaGetLastError();
  return e != cudaSuccess ? e : sum_partials(red, (int)blocks, 1, out, nullptr, s);
}

// F *= 1 / *denom
__global__ void k_scale_by_inv(float* F, int64_t total, const double* denom,
                               const DevStatus* gate) {
  if (gated_off(gate)) return;
  const float f = (float)(1.0 / *denom);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x)
    F[i] *= f;
}

cudaError_t launch_scale_by_inv(float* F, int64_t d, const double* denom, cudaStream_t s) {
  const int64_t tot = d * d;
  const int64_t blocks = std::min<int64_t>((tot + 255) / 256, (int64_t)num_sms() * 16);
  k_scale_by_inv<<<(unsigned)std::max<int64_t>(1, blocks), 256, 0, s>>>(F, tot, denom,
                                                                         current_gate());
  note_launches(1);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// the on-device convergence test and the stopped-fit bookkeeping
// ---------------------------------------------------------------------------
__global__ void k_copy_f64(double* dst, const double* src, const DevStatus* gate) {
  if (gated_off(gate)) return;
  *dst = *src;
}

cudaError_t launch_copy_f64(double* dst, const double* src, cudaStream_t s) {
  k_copy_f64<<<1, 1, 0, s>>>(dst, src, current_gate());
  note_launches(1);
  return cudaGetLastError();
}

__global__ void k_zero_f32(float* p, int64_t n, const DevStatus* gate) {
  if (gated_off(gate)) return;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    p[i] = 0.f;
}

cudaError_t launch_zero_f32(float* p, int64_t n, const DevStatus* gate, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const int64_t blocks = std::min<int64_t>((n + 255) / 256, (int64_t)num_sms() * 4);
  k_zero_f32<<<(unsigned)blocks, 256, 0, s>>>(p, n, gate);
  note_launches(1);
  return cudaGetLastError();
}

// One thread.  delta_t as in the fit's definition (Frobenius distance of the
// trace-normalised iterates relative to the new one, the larger of A and B); the record
// holds the squared distances and norms accumulated by k_delta.
__global__ void k_iter_end(DevStatus* st, const IterRecord* R, int t, float tol, int slot) {
  if (halted(st)) return;
  st->iters_done = t;
  st->slot = slot;
  if (tol > 0.f && t > 1) {
    const double dA = R->nA2 > 0.0 ? sqrt(R->dA2 / R->nA2) : 0.0;
    const double dB = R->nB2 > 0.0 ? sqrt(R->dB2 / R->nB2) : 0.0;
    if (fmax(dA, dB) < (double)tol) st->stop = 1;
  }
}

cudaError_t launch_iter_end(DevStatus* st, const IterRecord* R, int t, float tol, int slot,
                            cudaStream_t s) {
  k_iter_end<<<1, 1, 0, s>>>(st, R, t, tol, slot);
  note_launches(1);
  return cudaGetLastError();
}

__global__ void k_resume(DevStatus* st) { st->stop = 0; }

cudaError_t launch_resume(DevStatus* st, cudaStream_t s) {
  k_resume<<<1, 1, 0, s>>>(st);
  note_launches(1);
  return cudaGetLastError();
}

__global__ void k_select_copy(const DevStatus* st, const float* __restrict__ src0,
                              const float* __restrict__ src1, float* __restrict__ dst,
                              int64_t count) {
  const float* src = st->slot ? src1 : src0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count;
       i += (int64_t)gridDim.x * blockDim.x)
    dst[i] = src[i];
}

cudaError_t launch_select_copy(const DevStatus* st, const float* src0, const float* src1,
                               float* dst, int64_t count, cudaStream_t s) {
  if (count <= 0) return cudaSuccess;
  const int64_t blocks = std::min<int64_t>((count + 255) / 256, (int64_t)num_sms() * 8);
  k_select_copy<<<(unsigned)blocks, 256, 0, s>>>(st, src0, src1, dst, count);
  note_launches(1);
  return cudaGetLastError();
}

__global__ void k_record_at_done(const DevStatus* st, IterRecord* recs, size_t off,
                                 const double* src) {
  char* rec = reinterpret_cast<char*>(recs + st->iters_done);
  *reinterpret_cast<double*>(rec + off) = *src;
}

cudaError_t launch_record_at_done(const DevStatus* st, IterRecord* recs, size_t off,
                                  const double* src, cudaStream_t s) {
  k_record_at_done<<<1, 1, 0, s>>>(st, recs, off, src);
  note_launches(1);
  return cudaGetLastError();
}

// dst = scale * src (count floats; the product in fp64, one rounding)
__global__ void k_scale_copy(const float* __restrict__ src, float* __restrict__ dst,
                             int64_t count, double scale, const DevStatus* gate) {
  if (gated_off(gate)) return;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count;
       i += (int64_t)gridDim.x * blockDim.x)
    dst[i] = (float)((double)src[i] * scale);
}

cudaError_t launch_scale_copy(const float* src, float* dst, int64_t count, double scale,
                              cudaStream_t s) {
  if (count <= 0) return cudaSuccess;
  const int64_t blocks = std::min<int64_t>((count + 255) / 256, (int64_t)num_sms() * 8);
  k_scale_copy<<<(unsigned)blocks, 256, 0, s>>>(src, dst, count, scale, current_gate());
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace ffh
