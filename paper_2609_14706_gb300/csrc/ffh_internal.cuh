// Internal declarations shared by the libffh translation units.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "../../include/ffh.h"

namespace ffh {

// ---------------------------------------------------------------------------
// per-device one-time set-up
// ---------------------------------------------------------------------------
// A kernel's dynamic shared-memory limit is an attribute of the current device's
// context, so it is raised once per device, not once per process.  Bit i of `bits`
// records device i (safe to read and set from several host threads; devices >= 64
// repeat the set-up on every call, which is correct, only slower).
struct PerDeviceOnce {
  std::atomic<unsigned long long> bits{0};
  bool done(int dev) const {
    return dev >= 0 && dev < 64 && ((bits.load(std::memory_order_acquire) >> dev) & 1ull);
  }
  void set(int dev) {
    if (dev >= 0 && dev < 64) bits.fetch_or(1ull << dev, std::memory_order_acq_rel);
  }
};

// cudaFuncAttributeMaxDynamicSharedMemorySize = bytes for `func` on the current device,
// once per device (two threads may both set it the first time: same value, harmless).
inline cudaError_t smem_attr_once(const void* func, int bytes, PerDeviceOnce& once) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (once.done(dev)) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) once.set(dev);
  return e;
}

// ---------------------------------------------------------------------------
// device status block (one per handle, in the workspace)
// ---------------------------------------------------------------------------
struct DevStatus {
  int error;        // first FFH_ERR_* raised by a kernel (0 = none)
  int error_info;   // where: pivot index, or timeout site
  int abort_all;    // set together with error; kernels test it on entry
  int stop;         // the fit met its tolerance: the later iterations' kernels return at once
  double logdet;    // log|F| of the last Cholesky
  double acc[8];    // scratch reductions (traces, norms, dot products)
  int iters_done;   // iterations completed (written by the end-of-iteration kernel)
  int slot;         // ping-pong slot holding the last completed iterate (A and B)
  int pad[2];
};

// true once a kernel raised an error or the fit stopped at its tolerance: the kernels of
// a fit test this on entry (block-uniform) and return at once
__device__ __forceinline__ bool halted(const DevStatus* st) {
  return (*reinterpret_cast<const volatile int*>(&st->abort_all) |
          *reinterpret_cast<const volatile int*>(&st->stop)) != 0;
}
// Block-uniform gate test for the entry of a kernel (every thread of the block must call
// it): thread 0 reads the status and broadcasts it, so the block returns as a whole even
// if another stream's kernel raises an error meanwhile.
__device__ __forceinline__ bool gated_off(const DevStatus* gate) {
  if (gate == nullptr) return false;
  __shared__ int s_gated_off;
  if (threadIdx.x == 0 && threadIdx.y == 0 && threadIdx.z == 0) s_gated_off = halted(gate) ? 1 : 0;
  __syncthreads();
  return s_gated_off != 0;
}

// The status block of the fit that is being enqueued by this host thread (a handle is
// used by one thread at a time), or null.  Launchers of the small kernels pass it to
// their kernels, which then do nothing once that fit has stopped or failed.  Set for the
// duration of a fit by GateScope.
const DevStatus* current_gate();
void set_current_gate(const DevStatus* st);
struct GateScope {
  explicit GateScope(const DevStatus* st) { set_current_gate(st); }
  ~GateScope() { set_current_gate(nullptr); }
  GateScope(const GateScope&) = delete;
  GateScope& operator=(const GateScope&) = delete;
};

// per-iteration record kept on the device, read once at the end of a fit
struct IterRecord {
  double logdet_A_prev;  // log|A_{t-1}| (after normalisation)
  double logdet_B;       // log|B_t| before the A-side rescale
  double sum_qr_B;       // sum_k q_k r_k at (A_{t-1}, B_t)
  double sum_qr_A;       // sum_k q_k r_k at (A_t, B_t) (filled by the next iteration)
  double logdet_A;       // log|A_t| (filled by the next iteration)
  double scale;          // s = tr(A_t)/n before normalisation
  double dA2, nA2;       // ||A^_t - A^_{t-1}||^2, ||A^_t||^2
  double dB2, nB2;       // same for B
  double trB;            // tr(B_t) after the rescale
  double shift_B;        // damping shift added to B_t (0 undamped)
  double shift_A;        // damping shift added to A_t before the rescale
  double trinvB;         // tr(B_t^-1) = ||L_B^-1||_F^2 (matrix-sample fit)
  double trinvA;         // tr(A_t^-1) after the rescale (filled by the next iteration)
};

__device__ __forceinline__ void raise_error(DevStatus* st, int code, int info) {
  if (atomicCAS(&st->error, 0, code) == 0) {
    st->error_info = info;
  }
  atomicExch(&st->abort_all, 1);
}

// ---------------------------------------------------------------------------
// launch helpers (host)
// ---------------------------------------------------------------------------
struct Ctx;  // defined in ffh_api.cu

int num_sms();
// process-wide count of kernels launched by libffh
void note_launches(int k);
long long launches_so_far();

// tensor-core kernels (kernels_tc.cu)
// weighted-Gram output tile (rows x cols); a tile is computed iff it meets the lower
// triangle: tile_col * kGramBN <= tile_row * kGramBM + kGramBM - 1
constexpr int kGramBM = 256;
constexpr int kGramBN = 256;
constexpr int kGramBK = 64;   // samples per pipeline stage (weights padded to this)
// The Gram tile table: the tiles that meet the lower triangle, listed by square supertiles
// of kGramSuper x kGramSuper tiles (row-major over the supertiles of the lower triangle,
// row-major inside each).  The persistent CTAs take consecutive units, so one wave of CTAs
// covers about one supertile: its tiles share few operand feature blocks, which the CTAs
// stream through L2 at about the same sample position.  lut[ti * nbn + tj] = the tile's
// index, or -1 for tiles above the triangle.  Returns the tile count.
constexpr int kGramSuper = 12;
// Tile t of a row-major lower triangle of tiles: t = tm (tm + 1) / 2 + tn with tn <= tm (the
// float square root gives a first guess, the integer steps make it exact).
__host__ __device__ inline void lower_tile(int t, int& tm, int& tn) {
  int r = (int)((sqrtf(8.f * (float)t + 1.f) - 1.f) * 0.5f);
  while ((r + 1) * (r + 2) / 2 <= t) ++r;
  while (r * (r + 1) / 2 > t) --r;
  tm = r;
  tn = t - r * (r + 1) / 2;
}
__host__ __device__ inline int gram_fill_tiles(int nbm, int nbn, int2* tiles, int* lut) {
  int T = 0;
  for (int I = 0; I < nbm; I += kGramSuper)
    for (int J = 0; J < nbn && J <= I + kGramSuper - 1; J += kGramSuper)
      for (int ti = I; ti < nbm && ti < I + kGramSuper; ++ti)
        for (int tj = J; tj < nbn && tj < J + kGramSuper; ++tj) {
          // tile meets the lower triangle iff its first column <= its last row
          const bool need = (int64_t)tj * kGramBN <= (int64_t)ti * kGramBM + kGramBM - 1;
          if (need) {
            lut[ti * nbn + tj] = T;
            tiles[T++] = make_int2(ti, tj);
          }
        }
  for (int ti = 0; ti < nbm; ++ti)
    for (int tj = 0; tj < nbn; ++tj)
      if (!((int64_t)tj * kGramBN <= (int64_t)ti * kGramBM + kGramBM - 1)) lut[ti * nbn + tj] = -1;
  return T;
}
struct GramPlan {
  int T;        // lower-triangle output tiles
  int S;        // K splits
  int KB;       // kGramBK-sample blocks
  int units;    // T * S
  int grid;     // persistent CTAs
};
GramPlan gram_plan(int64_t N, int64_t d, int sms);
size_t gram_partial_bytes(const GramPlan& p);
// C = scale * V^T diag(w) V (lower tiles, then mirrored), V bf16 N x d (pitch ld elements).
// w_padded (nullable: w = 1) must be readable up to KB * kGramBK entries, zero past N; with
// weights, d and ld are multiples of 8 and V is 16-byte aligned.  after_main, if given, is
// recorded between the main kernel and the reduction.
cudaError_t launch_gram_tc(const __nv_bfloat16* V, int64_t N, int64_t d, int64_t ld,
                           const float* w_padded, float scale, float* C, int64_t ldc,
                           float* partial, int2* tiles_dev, int* tile_lut_dev,
                           const GramPlan& plan, DevStatus* st, int fault, cudaStream_t s,
                           cudaEvent_t after_main = nullptr);
// CTAs that share one 128-sample row block of the quadratic form (each takes a snake-ordered
// share of the 256-wide column blocks): 1 below 4 column blocks, 2 below 24, then 4, which
// keeps the row blocks in flight within L2 at large d
inline int qform_groups(int64_t d) {
  const int64_t nc = (d + 255) / 256;
  return nc >= 24 ? 4 : (nc >= 4 ? 2 : 1);
}
// fp32 scratch of the quadratic form over N samples of width d: the per-group partial sums
// when more than two groups share a row block (added in a fixed order afterwards)
inline size_t qform_scratch_floats(int64_t N, int64_t d) {
  return qform_groups(d) > 2 ? (size_t)qform_groups(d) * (size_t)N : 0;
}
// q_k = ||M v_k||^2, V bf16 N x d (pitch ld), M bf16 d x d lower (pitch ldm); qpart: at
// least qform_scratch_floats(N, d) floats (may be null when that is 0)
cudaError_t launch_qform_tc(const __nv_bfloat16* V, int64_t N, int64_t d, int64_t ld,
                            const __nv_bfloat16* M, int64_t ldm, float* q, float* qpart,
                            DevStatus* st, cudaStream_t s, bool upper = false);
// fp32 -> bf16 of the transpose of a lower-triangular matrix (upper result, zeros below)
cudaError_t launch_lowerT_to_bf16(const float* src, int64_t d, int64_t lds, __nv_bfloat16* dst,
                                  int64_t ldd, cudaStream_t s);
size_t gram_tile_table_bytes(int64_t d);
void gram_build_tiles(int64_t d, int2* tiles_host, int* lut_host, int* T_out);

// small CUDA-core kernels (kernels_simt.cu)
cudaError_t launch_rowsumsq(const void* V, int dtype, int64_t N, int64_t d, int64_t ld, float* q,
                            cudaStream_t s);
cudaError_t launch_to_bf16(const float* src, int64_t rows, int64_t cols, int64_t lds,
                           __nv_bfloat16* dst, int64_t ldd, cudaStream_t s);
// Streams and events of the look-ahead schedule of the tensor-core Cholesky: the panel
// chain (diagonal block, panel solve, update of the next column block) runs on `crit`
// (highest priority), the rest of each trailing update on `side` (lowest priority).
struct CholStreams {
  cudaStream_t crit = nullptr, side = nullptr;
  cudaEvent_t ev[5] = {};  // fork, panel solve done, trailing update done (x2), join
};
cudaError_t chol_streams_init(CholStreams* cs);
void chol_streams_destroy(CholStreams* cs);
// tensor-core Cholesky + inverse (kernels_chol.cu); `work` of cholesky_tc_work_bytes(d).
// With cs the work forks from s onto cs->crit / cs->side and joins back into s.
cudaError_t launch_cholesky_tc(const float* F, int64_t d, int64_t ldf, float* L, float* Linv,
                               void* work, DevStatus* st, int fault, cudaStream_t s,
                               CholStreams* cs = nullptr);
size_t cholesky_tc_work_bytes(int64_t d);
cudaError_t launch_fill_identity(float* F, int64_t d, int64_t ld, cudaStream_t s);

// WaterKron downstream (waterkron.cu)
cudaError_t launch_reverse_sym(const float* F, int64_t d, int64_t ldf, float* out, cudaStream_t s);
cudaError_t launch_rev_transpose(const float* C, int64_t d, float* out, bool normalize,
                                 cudaStream_t s);
cudaError_t launch_waterfilling(const float* LA, int64_t n, const float* LB, int64_t m,
                                float gamma, float* alpha, float* beta, cudaStream_t s);
size_t gptq2_work_bytes(int64_t m, int64_t n);
cudaError_t launch_gptq2(const float* W, const float* LtA, const float* LtB, const float* alpha,
                         const float* beta, int64_t m, int64_t n, int32_t* Z, float* V,
                         void* work, DevStatus* st, cudaStream_t s);
cudaError_t launch_damp(float* F, int64_t d, int64_t ld, float lambda, DevStatus* st,
                        cudaStream_t s, double* shift_out = nullptr);
cudaError_t launch_add(float* C, const float* X, int64_t total, cudaStream_t s);
// matrix samples (kernels_matrix.cu): V rows (k, r) = (M Gop_k)[r][:], see the file
cudaError_t launch_transform_tc(const __nv_bfloat16* M, int64_t d, int64_t ldm,
                                const __nv_bfloat16* Gb, int64_t nk, int64_t m, int64_t n,
                                bool b_update, __nv_bfloat16* V, DevStatus* st, cudaStream_t s);
// A <- A / s, B <- B * s with s = tr(A)/n; records s and log-determinant corrections
cudaError_t launch_normalize(float* A, int64_t n, float* B, int64_t m, IterRecord* rec,
                             DevStatus* st, cudaStream_t s);
// fp64 reductions write per-block partial sums to a scratch of kRedDoubles doubles and add
// them in a fixed order (bit-reproducible statistics)
constexpr int kRedDoubles = 4096;
cudaError_t launch_delta(const float* F, const float* Fprev, int64_t d, double* d2, double* n2,
                         double* tr, double* red, cudaStream_t s);
cudaError_t launch_dot(const float* a, const float* b, int64_t N, double* out, double* red,
                       cudaStream_t s);
cudaError_t launch_frob2(const float* F, int64_t d, double* out, double* red, cudaStream_t s);
cudaError_t launch_scale_by_inv(float* F, int64_t d, const double* denom, cudaStream_t s);
// dst = scale * src
cudaError_t launch_scale_copy(const float* src, float* dst, int64_t count, double scale,
                              cudaStream_t s);
// *dst = *src (fp64 record fields; gated like the other small kernels)
cudaError_t launch_copy_f64(double* dst, const double* src, cudaStream_t s);
// fp32 zero fill, skipped once `gate` has stopped or failed (gate may be null)
cudaError_t launch_zero_f32(float* p, int64_t n, const DevStatus* gate, cudaStream_t s);
// end of iteration t: unless the fit has stopped, record t and the slot of its iterate,
// and with tol > 0 and t > 1 set st->stop when delta_t = max(sqrt(dA2/nA2),
// sqrt(dB2/nB2)) of record R is below tol
cudaError_t launch_iter_end(DevStatus* st, const IterRecord* R, int t, float tol, int slot,
                            cudaStream_t s);
// clear st->stop (the evaluation after a stopped fit runs again)
cudaError_t launch_resume(DevStatus* st, cudaStream_t s);
// dst = (st->slot ? src1 : src0), count floats
cudaError_t launch_select_copy(const DevStatus* st, const float* src0, const float* src1,
                               float* dst, int64_t count, cudaStream_t s);
// recs[st->iters_done].<field at byte offset off> = *src
cudaError_t launch_record_at_done(const DevStatus* st, IterRecord* recs, size_t off,
                                  const double* src, cudaStream_t s);

}  // namespace ffh
