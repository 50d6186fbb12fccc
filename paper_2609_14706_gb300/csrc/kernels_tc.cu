// Tensor-core (tcgen05 + TMA + TMEM) kernels of the FlipFlop Hessian fit:
//
//  * k_gram_tc   -- weighted Gram  C = scale * V^T diag(w) V  (the E[w v v^T] of the
//                   Section 5 updates).  V is N x d bf16, row-major (one sample per row),
//                   so both MMA operands are the same V read "MN-major": TMA boxes of
//                   64 features x 64 samples, 128-byte swizzle.  diag(w) is applied to the
//                   A operand in shared memory between the TMA landing and the MMA (one
//                   16-byte vector = 8 features of one sample share one weight), so no
//                   scaled copy of V exists anywhere.  Only the tiles that meet the lower
//                   triangle are computed; K (samples) is split into S slices so that
//                   tiles x slices fill the SMs; fp32 partial tiles go to a workspace and
//                   k_gram_reduce sums them in a fixed order, applies the scale and writes
//                   both triangles.
//  * k_qform_tc  -- q_k = ||M v_k||^2 for lower-triangular M = L^-1 (the x^T A^-1 x of
//                   Section 5).  Y = V M^T is formed tile by tile in TMEM and squared and
//                   row-summed by the epilogue straight from TMEM, so Y never reaches
//                   HBM.  Column block c of Y only needs K < 256 (c+1) (M is lower); an
//                   upper-triangular M (the Frobenius variant's x^T A x = ||L^T x||^2)
//                   needs K >= 256 c only.
//
// Both are persistent (one CTA per SM, warp-specialised): warp 0 issues TMA, warp 1
// issues tcgen05.mma, warp 2 owns the TMEM allocation, warps 4-7 stage / drain.
// Every mbarrier wait is bounded; on expiry the kernel records FFH_ERR_TIMEOUT,
// drains what it issued and returns.
#include <cudaTypedefs.h>

#include <algorithm>
#include <vector>

#include "ffh_internal.cuh"
#include "tc_ptx.cuh"

namespace ffh {

using namespace ptx;

static constexpr uint64_t kWaitBudgetNs = 4000000000ull;      // 4 s
static constexpr uint64_t kFaultWaitBudgetNs = 20000000ull;   // 20 ms (fault injection)

// ---------------------------------------------------------------------------
// tensor maps
// ---------------------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  // the driver entry point is the same for every device; looked up once, thread-safely
  static const PFN_cuTensorMapEncodeTiled_v12000 fn = []() {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    return (PFN_cuTensorMapEncodeTiled_v12000) nullptr;
  }();
  return fn;
}

// 2-D bf16 map: inner extent `inner` elements (contiguous), `outer` rows of pitch
// `pitch_elems`; box box_inner x box_outer; 128-byte swizzle; out-of-range reads as 0.
static bool make_map_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                          uint64_t pitch_elems, uint32_t box_inner, uint32_t box_outer) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {pitch_elems * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t es[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

__device__ __forceinline__ uint32_t scale_bf16x2(uint32_t v, float s) {
  float lo = __uint_as_float(v << 16) * s;
  float hi = __uint_as_float(v & 0xFFFF0000u) * s;
  __nv_bfloat162 r = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&r);
}

// ===========================================================================
// weighted Gram
// ===========================================================================
namespace gram {
constexpr int BM = kGramBM;  // output rows (features i) per tile: two M = 128 MMAs
constexpr int BN = kGramBN;  // output cols (features j) per tile
constexpr int BK = kGramBK;  // samples per pipeline stage
constexpr int STAGES = 3;    // 3 x 64 KB: fewer, larger stages keep the MMA fed
constexpr int BOX_BYTES = 64 * BK * 2;  // one TMA box: 64 features x BK samples
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr uint32_t TMEM_COLS = 512;     // two 128 x 256 fp32 accumulators
constexpr int THREADS = 384;            // warps 0-3: TMA, MMA, TMEM; warps 4-11: scale + drain
constexpr int NSCALE = THREADS - 128;
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + STAGES * BK * 4 + 256;
}  // namespace gram

struct GramArgs {
  const float* w;        // weights padded with zeros to KB*BK, or nullptr (w = 1)
  float* partial;        // [units][BN][BM] fp32
  const int2* tiles;     // T lower-triangle tiles (tile row, tile col)
  int T, S, KB, units;
  DevStatus* st;
  int fault;
  unsigned long long budget_ns;
};

__global__ void __launch_bounds__(gram::THREADS, 1)
    k_gram_tc(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap bmap,
              const GramArgs a) {
  using namespace gram;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* stages = smem;
  float* wbuf = reinterpret_cast<float*>(smem + STAGES * STAGE_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(wbuf + STAGES * BK);
  uint64_t* full = bars;
  uint64_t* scaled = bars + STAGES;
  uint64_t* empty = bars + 2 * STAGES;
  uint64_t* accf = bars + 3 * STAGES;
  uint64_t* acce = accf + 1;
  uint64_t* drain = acce + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* skip_flag = abort_flag + 1;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    *skip_flag = halted(a.st) ? 1 : 0;
    *abort_flag = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&scaled[s], NSCALE);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accf, 1);
    mbar_init(acce, NSCALE);
    mbar_init(drain, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (*skip_flag) return;  // an earlier step failed: do nothing (block-uniform)
  if (warp == 2) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&amap);
    prefetch_tmap(&bmap);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint64_t budget = a.budget_ns;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      uint32_t it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < a.units && ok; u += gridDim.x) {
        const int split = u / a.T, tile = u - split * a.T;
        const int2 tt = a.tiles[tile];
        const int kb0 = static_cast<int>((int64_t)a.KB * split / a.S);
        const int kb1 = static_cast<int>((int64_t)a.KB * (split + 1) / a.S);
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, budget)) {
            ok = false;
            break;
          }
          const bool drop = (a.fault == FFH_FAULT_LOST_COPY) && blockIdx.x == 0 && it == 2;
          mbar_arrive_expect_tx(&full[s], STAGE_BYTES + (a.w ? BK * 4 : 0));
          if (!drop) {
            uint8_t* sa = stages + s * STAGE_BYTES;
            uint8_t* sb = sa + A_BYTES;
            const int y = kb * BK;
#pragma unroll
            for (int c = 0; c < BM / 64; ++c)
              tma_load_2d(sa + c * BOX_BYTES, &amap, &full[s], tt.x * BM + c * 64, y);
#pragma unroll
            for (int c = 0; c < BN / 64; ++c)
              tma_load_2d(sb + c * BOX_BYTES, &bmap, &full[s], tt.y * BN + c * 64, y);
            if (a.w) bulk_load(wbuf + s * BK, a.w + (size_t)kb * BK, BK * 4, &full[s]);
          }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        raise_error(a.st, FFH_ERR_TIMEOUT, 1);
      }
      // drain: every copy this thread issued must land before the CTA exits
      const uint32_t first = it > STAGES ? it - STAGES : 0;
      for (uint32_t j = first; j < it; ++j) {
        volatile int never = 0;
        mbar_wait(&full[j % STAGES], (j / STAGES) & 1, &never,
                  a.fault ? kFaultWaitBudgetNs : budget);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      constexpr uint32_t idesc = idesc_bf16_f32(128, BN, true, true);
      uint32_t it = 0, acc_ph = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < a.units && ok; u += gridDim.x) {
        const int split = u / a.T;
        const int kb0 = static_cast<int>((int64_t)a.KB * split / a.S);
        const int kb1 = static_cast<int>((int64_t)a.KB * (split + 1) / a.S);
        if (!mbar_wait(acce, acc_ph ^ 1, abort_flag, budget)) {
          ok = false;
          break;
        }
        tc_fence_after();
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          // unweighted: the operands are ready when the TMA lands; weighted: when the
          // staging warps have scaled A
          if (!mbar_wait(a.w ? &scaled[s] : &full[s], ph, abort_flag, budget)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(stages + s * STAGE_BYTES);
          const uint32_t sb = sa + A_BYTES;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            // MN-major, 128B swizzle: 16 samples = two 8-row groups (1024 B each);
            // 64-feature blocks are one TMA box (BOX_BYTES) apart.
            const uint64_t bd = sw128_desc(sb + k * 2048, BOX_BYTES, 1024);
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
              const uint64_t ad = sw128_desc(sa + hh * 2 * BOX_BYTES + k * 2048, BOX_BYTES, 1024);
              mma_bf16(tmem + hh * BN, ad, bd, idesc, (kb > kb0 || k > 0) ? 1u : 0u);
            }
          }
          mma_commit(&empty[s]);
        }
        if (!ok) break;
        mma_commit(accf);
        acc_ph ^= 1;
      }
      if (!ok) {
        *abort_flag = 1;
        raise_error(a.st, FFH_ERR_TIMEOUT, 2);
      }
      // drain: wait for every MMA issued by this thread
      mma_commit(drain);
      volatile int never = 0;
      mbar_wait(drain, 0, &never, a.fault ? kFaultWaitBudgetNs : budget);
    }
  } else if (warp >= 4) {
    // ---------------- weight staging + epilogue ----------------
    const int t = threadIdx.x - 128;
    const int wq = warp & 3;          // TMEM lanes 32*wq .. 32*wq+31
    const int hh = (warp - 4) >> 2;   // accumulator (tile rows 128*hh ..)
    uint32_t it = 0, acc_ph = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < a.units && ok; u += gridDim.x) {
      const int split = u / a.T;
      const int kb0 = static_cast<int>((int64_t)a.KB * split / a.S);
      const int kb1 = static_cast<int>((int64_t)a.KB * (split + 1) / a.S);
      for (int kb = kb0; kb < kb1 && a.w; ++kb, ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1;
        if (!mbar_wait(&full[s], ph, abort_flag, a.fault ? kFaultWaitBudgetNs : budget)) {
          ok = false;
          break;
        }
        {
          uint4* A4 = reinterpret_cast<uint4*>(stages + s * STAGE_BYTES);
          const float* wr = wbuf + s * BK;
          constexpr int CHUNKS_PER_BOX = BOX_BYTES / 16;
#pragma unroll
          for (int c = t; c < A_BYTES / 16; c += NSCALE) {
            // 16-byte chunk c: sample (row of its box) = (c % CHUNKS_PER_BOX) / 8; the
            // swizzle only permutes chunks within a 128-byte row.
            const float wv = wr[(c & (CHUNKS_PER_BOX - 1)) >> 3];
            uint4 v = A4[c];
            v.x = scale_bf16x2(v.x, wv);
            v.y = scale_bf16x2(v.y, wv);
            v.z = scale_bf16x2(v.z, wv);
            v.w = scale_bf16x2(v.w, wv);
            A4[c] = v;
          }
          fence_proxy_async_smem();
        }
        mbar_arrive(&scaled[s]);
      }
      if (!ok) break;
      if (!mbar_wait(accf, acc_ph, abort_flag, budget)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float* out = a.partial + (size_t)u * (BN * BM);
      const int row = hh * 128 + wq * 32 + lane;
#pragma unroll 1
      for (int cb = 0; cb < BN / 32; ++cb) {
        float v[32];
        tmem_ld32(tmem + ((uint32_t)(wq * 32) << 16) + hh * BN + cb * 32, v);
#pragma unroll
        for (int j = 0; j < 32; ++j) out[(size_t)(cb * 32 + j) * BM + row] = v[j];
      }
      tc_fence_before();
      mbar_arrive(acce);
      acc_ph ^= 1;
    }
    if (!ok) {
      *abort_flag = 1;
      raise_error(a.st, FFH_ERR_TIMEOUT, 3);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// Sum the S partial tiles of each lower-triangle element in a fixed order, scale, and
// write C[i][j] and C[j][i].  Block = 32 x 8 threads over one 32 x 32 block.
__global__ void k_gram_reduce(const float* __restrict__ partial, const int* __restrict__ lut,
                              int nbn, int T, int S, int64_t d, float scale, float* C,
                              int64_t ldc, const DevStatus* gate) {
  using namespace gram;
  const int bi = blockIdx.y, bj = blockIdx.x;
  if (bj > bi) return;
  if (gated_off(gate)) return;
  __shared__ float tile[32][33];
  const int64_t i0 = (int64_t)bi * 32, j0 = (int64_t)bj * 32;
  const size_t split_stride = (size_t)T * BN * BM;
  for (int r = threadIdx.y; r < 32; r += 8) {
    const int64_t i = i0 + threadIdx.x, j = j0 + r;
    float v = 0.f;
    if (i < d && j < d && i >= j) {
      const int ti = (int)(i / BM), tj = (int)(j / BN);
      const int t = lut[ti * nbn + tj];
      const float* p = partial + ((size_t)t * BN + (size_t)(j - (int64_t)tj * BN)) * BM +
                       (size_t)(i - (int64_t)ti * BM);
      float acc = 0.f;
      for (int s = 0; s < S; ++s) acc += p[s * split_stride];
      v = acc * scale;
      C[j * ldc + i] = v;
    }
    tile[r][threadIdx.x] = v;
  }
  __syncthreads();
  for (int r = threadIdx.y; r < 32; r += 8) {
    const int64_t i = i0 + r, j = j0 + threadIdx.x;
    if (i < d && j < d && i >= j) C[i * ldc + j] = tile[threadIdx.x][r];
  }
}

size_t gram_tile_table_bytes(int64_t d) {
  const int64_t nbm = (d + gram::BM - 1) / gram::BM, nbn = (d + gram::BN - 1) / gram::BN;
  return (size_t)(nbm * nbn) * (sizeof(int2) + sizeof(int));
}

void gram_build_tiles(int64_t d, int2* tiles, int* lut, int* T_out) {
  const int nbm = (int)((d + gram::BM - 1) / gram::BM);
  const int nbn = (int)((d + gram::BN - 1) / gram::BN);
  *T_out = gram_fill_tiles(nbm, nbn, tiles, lut);
}

GramPlan gram_plan(int64_t N, int64_t d, int sms) {
  GramPlan p{};
  const int nbm = (int)((d + gram::BM - 1) / gram::BM);
  const int nbn = (int)((d + gram::BN - 1) / gram::BN);
  int T = 0;
  for (int ti = 0; ti < nbm; ++ti)
    for (int tj = 0; tj < nbn; ++tj)
      if ((int64_t)tj * gram::BN <= (int64_t)ti * gram::BM + gram::BM - 1) ++T;
  p.T = T;
  p.KB = (int)std::max<int64_t>(1, (N + gram::BK - 1) / gram::BK);
  // Split count.  (1) No unit sums more than kMaxUnitSamples samples into its fp32
  // accumulator: the error of one tensor-core accumulator over many MMAs grows with their
  // number (a fit's Kronecker error measured 1.6e-4 with 26K samples per accumulator and
  // 1.8e-3 with 262K).  (2) Among the counts that allow, fill the SMs with equal-size units
  // (wave efficiency), at least 16 blocks of samples per unit.  (3) The partial tiles stay
  // within kMaxPartialBytes (then (1) gives way).
  constexpr int64_t kMaxUnitSamples = 32768;
  constexpr double kMaxPartialBytes = 8.0e9;
  const double unit_bytes = (double)gram::BN * gram::BM * 4.0;
  const int s_acc = (int)((p.KB + kMaxUnitSamples / gram::BK - 1) / (kMaxUnitSamples / gram::BK));
  const int s_mem = std::max(1, (int)(kMaxPartialBytes / ((double)T * unit_bytes)));
  const int s_min = std::max(1, std::min(s_acc, s_mem));
  const int max_s = std::max(s_min, std::min(64, p.KB / 16));
  int best_s = s_min;
  double best_eff = -1.0;
  for (int s = s_min; s <= max_s; ++s) {
    if ((double)T * s * unit_bytes > kMaxPartialBytes && s > s_min) break;
    const int64_t units = (int64_t)T * s;
    const int64_t waves = (units + sms - 1) / sms;
    const double eff = (double)units / (double)(waves * sms);
    if (eff > best_eff + 0.02) {
      best_eff = eff;
      best_s = s;
    }
  }
  p.S = best_s;
  p.units = T * best_s;
  p.grid = std::min(p.units, sms);
  return p;
}

size_t gram_partial_bytes(const GramPlan& p) {
  return (size_t)p.units * gram::BN * gram::BM * sizeof(float);
}

cudaError_t launch_gram_tc(const __nv_bfloat16* V, int64_t N, int64_t d, int64_t ld,
                           const float* w_padded, float scale, float* C, int64_t ldc,
                           float* partial, int2* tiles_dev, int* lut_dev, const GramPlan& plan,
                           DevStatus* st, int fault, cudaStream_t s, cudaEvent_t after_main) {
  // the weights are bulk-copied 64 at a time (16-byte aligned source)
  if (w_padded && (reinterpret_cast<uintptr_t>(w_padded) & 15)) return cudaErrorInvalidValue;
  CUtensorMap map;
  if (!make_map_bf16(&map, V, (uint64_t)d, (uint64_t)N, (uint64_t)ld, 64, gram::BK))
    return cudaErrorInvalidValue;
  static PerDeviceOnce attr;
  {
    cudaError_t e = smem_attr_once((const void*)k_gram_tc, gram::SMEM_BYTES, attr);
    if (e != cudaSuccess) return e;
  }
  GramArgs a;
  a.w = w_padded;
  a.partial = partial;
  a.tiles = tiles_dev;
  a.T = plan.T;
  a.S = plan.S;
  a.KB = plan.KB;
  a.units = plan.units;
  a.st = st;
  a.fault = fault;
  a.budget_ns = fault == FFH_FAULT_LOST_COPY ? kFaultWaitBudgetNs : kWaitBudgetNs;
  k_gram_tc<<<plan.grid, gram::THREADS, gram::SMEM_BYTES, s>>>(map, map, a);
  note_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (after_main) {
    // a timing event: inside a stream capture it must become a graph node of its own
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if ((e = cudaStreamIsCapturing(s, &cap)) != cudaSuccess) return e;
    e = cap == cudaStreamCaptureStatusActive
            ? cudaEventRecordWithFlags(after_main, s, cudaEventRecordExternal)
            : cudaEventRecord(after_main, s);
    if (e != cudaSuccess) return e;
  }
  const int nb32 = (int)((d + 31) / 32);
  const int nbn = (int)((d + gram::BN - 1) / gram::BN);
  k_gram_reduce<<<dim3(nb32, nb32), dim3(32, 8), 0, s>>>(partial, lut_dev, nbn, plan.T, plan.S,
                                                         d, scale, C, ldc, st);
  note_launches(1);
  return cudaGetLastError();
}

// ===========================================================================
// fused quadratic form
// ===========================================================================
namespace qf {
constexpr int BM = 128;   // samples per row block
constexpr int BN = 256;   // output features per column block
constexpr int BK = 64;    // K (input features) per stage
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr uint32_t TMEM_COLS = 512;  // two 256-column accumulators
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + 256;
constexpr int THREADS = 256;
}  // namespace qf

// Group of column block c when G CTAs share a row block: the blocks are dealt out in a
// snake (0, 1, .., G-1, G-1, .., 1, 0, 0, 1, ..), which balances the triangular K ranges
// (block c costs c + 1 K-blocks of 256).
__host__ __device__ inline int qf_group(int c, int G) {
  const int p = c % (2 * G);
  return p < G ? p : 2 * G - 1 - p;
}

struct QformArgs {
  float* q;
  float* qpart;  // [G][N] per-group partial sums when G > 2
  int64_t N;
  int upper;  // M upper-triangular (column block c needs K >= 256 c) instead of lower
  int G;     // column-block groups per row block (qform_groups): G CTAs share a row block
             // (dividing the L2 working set by G); with 2 they add their sums into q (two
             // addends: order-independent), with more they write qpart, summed afterwards
  int RB;    // row blocks
  int NC;    // column blocks
  int KBd;   // 64-wide K blocks of d
  DevStatus* st;
  unsigned long long budget_ns;
};

__global__ void __launch_bounds__(qf::THREADS, 1)
    k_qform_tc(const __grid_constant__ CUtensorMap vmap, const __grid_constant__ CUtensorMap mmap,
               const QformArgs a) {
  using namespace qf;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* stages = smem;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;  // [2]
  uint64_t* acce = accf + 2;           // [2]
  uint64_t* drain = acce + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* skip_flag = abort_flag + 1;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    *skip_flag = halted(a.st) ? 1 : 0;
    *abort_flag = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], 128);
    }
    mbar_init(drain, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (*skip_flag) return;
  if (warp == 2) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&vmap);
    prefetch_tmap(&mmap);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint64_t budget = a.budget_ns;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < a.RB * a.G && ok; u += gridDim.x) {
        const int rb = u / a.G, grp = u - rb * a.G;
        for (int c = 0; c < a.NC && ok; ++c) {
          if (a.G > 1 && qf_group(c, a.G) != grp) continue;
          const int kb_lo = a.upper ? 4 * c : 0;
          const int kb_hi = a.upper ? a.KBd : min(a.KBd, 4 * (c + 1));
          for (int kb = kb_lo; kb < kb_hi; ++kb, ++it) {
            const int s = it % STAGES;
            const uint32_t ph = (it / STAGES) & 1;
            if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, budget)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&full[s], STAGE_BYTES);
            uint8_t* sa = stages + s * STAGE_BYTES;
            tma_load_2d(sa, &vmap, &full[s], kb * BK, rb * BM);
            tma_load_2d(sa + A_BYTES, &mmap, &full[s], kb * BK, c * BN);
          }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        raise_error(a.st, FFH_ERR_TIMEOUT, 11);
      }
      const uint32_t first = it > STAGES ? it - STAGES : 0;
      for (uint32_t j = first; j < it; ++j) {
        volatile int never = 0;
        mbar_wait(&full[j % STAGES], (j / STAGES) & 1, &never, budget);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, false, false);
      uint32_t it = 0, cc = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < a.RB * a.G && ok; u += gridDim.x) {
        const int grp = u % a.G;
        for (int c = 0; c < a.NC; ++c) {
          if (a.G > 1 && qf_group(c, a.G) != grp) continue;
          const int buf = cc & 1;
          if (!mbar_wait(&acce[buf], ((cc >> 1) & 1) ^ 1, abort_flag, budget)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int kb_lo = a.upper ? 4 * c : 0;
          const int kb_hi = a.upper ? a.KBd : min(a.KBd, 4 * (c + 1));
          for (int kb = kb_lo; kb < kb_hi; ++kb, ++it) {
            const int s = it % STAGES;
            const uint32_t ph = (it / STAGES) & 1;
            if (!mbar_wait(&full[s], ph, abort_flag, budget)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(stages + s * STAGE_BYTES);
            const uint32_t sb = sa + A_BYTES;
#pragma unroll
            for (int k = 0; k < BK / 16; ++k) {
              // K-major, 128B swizzle: rows of 128 B, 8-row groups 1024 B apart;
              // 16 K-elements = 32 B along the row.
              const uint64_t ad = sw128_desc(sa + k * 32, 16, 1024);
              const uint64_t bd = sw128_desc(sb + k * 32, 16, 1024);
              mma_bf16(tmem + buf * BN, ad, bd, idesc, (kb > kb_lo || k > 0) ? 1u : 0u);
            }
            mma_commit(&empty[s]);
          }
          if (!ok) break;
          mma_commit(&accf[buf]);
          ++cc;
        }
      }
      if (!ok) {
        *abort_flag = 1;
        raise_error(a.st, FFH_ERR_TIMEOUT, 12);
      }
      mma_commit(drain);
      volatile int never = 0;
      mbar_wait(drain, 0, &never, budget);
    }
  } else if (warp >= 4) {
    const int wq = warp - 4;
    uint32_t cc = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < a.RB * a.G && ok; u += gridDim.x) {
      const int rb = u / a.G, grp = u - rb * a.G;
      float acc = 0.f;
      for (int c = 0; c < a.NC; ++c) {
        if (a.G > 1 && qf_group(c, a.G) != grp) continue;
        const int buf = cc & 1;
        const uint32_t aph = (cc >> 1) & 1;
        ++cc;
        if (!mbar_wait(&accf[buf], aph, abort_flag, budget)) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll 1
        for (int cb = 0; cb < BN / 32; ++cb) {
          float v[32];
          tmem_ld32(tmem + ((uint32_t)(wq * 32) << 16) + buf * BN + cb * 32, v);
#pragma unroll
          for (int j = 0; j < 32; ++j) acc = fmaf(v[j], v[j], acc);
        }
        tc_fence_before();
        mbar_arrive(&acce[buf]);
      }
      if (!ok) break;
      const int64_t row = (int64_t)rb * BM + wq * 32 + lane;
      // two groups: q was zeroed and receives exactly two addends (order-independent)
      if (row < a.N) {
        if (a.G > 2)
          a.qpart[(int64_t)grp * a.N + row] = acc;
        else if (a.G == 2)
          atomicAdd(&a.q[row], acc);
        else
          a.q[row] = acc;
      }
    }
    if (!ok) {
      *abort_flag = 1;
      raise_error(a.st, FFH_ERR_TIMEOUT, 13);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// q_k = sum over the G groups of the partial sums, in group order (bit-reproducible)
__global__ void k_qform_sum(const float* __restrict__ qpart, int G, int64_t N, float* q,
                            const DevStatus* gate) {
  if (gated_off(gate)) return;
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < N;
       k += (int64_t)gridDim.x * blockDim.x) {
    float acc = qpart[k];
    for (int g = 1; g < G; ++g) acc += qpart[(int64_t)g * N + k];
    q[k] = acc;
  }
}

cudaError_t launch_qform_tc(const __nv_bfloat16* V, int64_t N, int64_t d, int64_t ld,
                            const __nv_bfloat16* M, int64_t ldm, float* q, float* qpart,
                            DevStatus* st, cudaStream_t s, bool upper) {
  CUtensorMap vmap, mmap;
  if (!make_map_bf16(&vmap, V, (uint64_t)d, (uint64_t)N, (uint64_t)ld, qf::BK, qf::BM))
    return cudaErrorInvalidValue;
  if (!make_map_bf16(&mmap, M, (uint64_t)d, (uint64_t)d, (uint64_t)ldm, qf::BK, qf::BN))
    return cudaErrorInvalidValue;
  static PerDeviceOnce attr;
  {
    cudaError_t e = smem_attr_once((const void*)k_qform_tc, qf::SMEM_BYTES, attr);
    if (e != cudaSuccess) return e;
  }
  QformArgs a;
  a.q = q;
  a.qpart = qpart;
  a.N = N;
  a.upper = upper ? 1 : 0;
  a.RB = (int)((N + qf::BM - 1) / qf::BM);
  a.NC = (int)((d + qf::BN - 1) / qf::BN);
  a.G = qform_groups(d);
  if (a.G > 2 && !qpart) return cudaErrorInvalidValue;
  a.KBd = (int)((d + qf::BK - 1) / qf::BK);
  a.st = st;
  a.budget_ns = kWaitBudgetNs;
  if (a.G == 2) {
    // the two groups add into q
    cudaError_t e = launch_zero_f32(q, N, st, s);
    if (e != cudaSuccess) return e;
  }
  const int grid = std::min(a.RB * a.G, num_sms());
  k_qform_tc<<<grid, qf::THREADS, qf::SMEM_BYTES, s>>>(vmap, mmap, a);
  note_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || a.G <= 2) return e;
  const int64_t blocks = std::min<int64_t>((N + 255) / 256, (int64_t)num_sms() * 8);
  k_qform_sum<<<(unsigned)blocks, 256, 0, s>>>(qpart, a.G, N, q, st);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace ffh
