// Matrix-sample transform for the FlipFlop fit to general samples G_k in R^{m x n}
// (Section 5, first form of each update):
//   B-update: B = 1/(N n) sum_k G_k A^-1 G_k^T = 1/(N n) sum_k Z_k Z_k^T,
//             Z_k^T = M_A G_k^T  (n x m),  M_A = chol(A)^-1;
//   A-update: A = 1/(N m) sum_k G_k^T B^-1 G_k = 1/(N m) sum_k Y_k^T Y_k,
//             Y_k = M_B G_k      (m x n),  M_B = chol(B)^-1.
// Both are "lower-triangular M times each sample", written as bf16 rows of a tall
// matrix V (rows (k, r)), whose unweighted Gram V^T V is the update.
//
// k_transform_tc: persistent tcgen05 kernel over units (sample k, row tile, col tile):
//   D[r][c] = sum_j M[r][j] Gop_k[j][c], with
//     KMAJOR (B-update): Gop_k[j][c] = G_k[c][j]  (G_k rows are the K-major B operand)
//     MN     (A-update): Gop_k[j][c] = G_k[j][c]  (G_k rows give an MN-major B operand)
//   M lower-triangular: row tile r0 needs K < r0 + 128 only.  Two TMEM accumulators
//   let the bf16 epilogue of one unit overlap the MMAs of the next.
#include <cudaTypedefs.h>

#include <algorithm>

#include "ffh_internal.cuh"
#include "tc_ptx.cuh"

namespace ffh {

using namespace ptx;

static constexpr uint64_t kTfWaitNs = 4000000000ull;

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn_mx() {
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

static bool map2d_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows,
                       uint64_t pitch_elems, uint32_t box_inner, uint32_t box_rows) {
  auto fn = encode_fn_mx();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {pitch_elems * 2};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace tf {
constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2, B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int BOX_MN_BYTES = 64 * BK * 2;  // MN-major B box: 64 columns x 64 K rows
constexpr uint32_t TMEM_COLS = 512;
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + 256;
constexpr int THREADS = 256;
}  // namespace tf

struct TransformArgs {
  __nv_bfloat16* V;  // output rows (k, r): row k*d_out + r, pitch ldv
  int64_t ldv;
  int d_out;         // rows of M (= d), rows per sample in V
  int d_other;       // columns of the output
  int d_in;          // K extent (= d)
  int g_rows;        // rows per sample in the 2-D view of G (m)
  int nk;            // samples in this launch
  int RT, CT;        // row / column tiles per sample
  int units;
  DevStatus* st;
};

template <bool MN>
__global__ void __launch_bounds__(tf::THREADS, 1)
    k_transform_tc(const __grid_constant__ CUtensorMap mmap, const __grid_constant__ CUtensorMap gmap,
                   const TransformArgs a) {
  using namespace tf;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
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
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int per_k = a.RT * a.CT;
  const int KB = (a.d_in + BK - 1) / BK;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < a.units && ok; u += gridDim.x) {
        const int k = u / per_k, rem = u - k * per_k;
        const int rt = rem / a.CT, ct = rem - rt * a.CT;
        const int nkb = min(KB, (rt * BM + BM + BK - 1) / BK);
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, kTfWaitNs)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], STAGE_BYTES);
          uint8_t* sa = smem + s * STAGE_BYTES;
          tma_load_2d(sa, &mmap, &full[s], kb * BK, rt * BM);
          if (!MN) {
            // rows c of G_k (output columns), K = j along the row
            tma_load_2d(sa + A_BYTES, &gmap, &full[s], kb * BK, k * a.g_rows + ct * BN);
          } else {
            // rows j of G_k (K), 64-column boxes of the output columns c
#pragma unroll
            for (int c = 0; c < BN / 64; ++c)
              tma_load_2d(sa + A_BYTES + c * BOX_MN_BYTES, &gmap, &full[s], ct * BN + c * 64,
                          k * a.g_rows + kb * BK);
          }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        raise_error(a.st, FFH_ERR_TIMEOUT, 31);
      }
      const uint32_t first = it > STAGES ? it - STAGES : 0;
      for (uint32_t j = first; j < it; ++j) {
        volatile int never = 0;
        mbar_wait(&full[j % STAGES], (j / STAGES) & 1, &never, kTfWaitNs);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, false, MN);
      uint32_t it = 0, cc = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < a.units && ok; u += gridDim.x, ++cc) {
        const int k = u / per_k, rem = u - k * per_k;
        const int rt = rem / a.CT;
        const int nkb = min(KB, (rt * BM + BM + BK - 1) / BK);
        const int buf = cc & 1;
        if (!mbar_wait(&acce[buf], ((cc >> 1) & 1) ^ 1, abort_flag, kTfWaitNs)) {
          ok = false;
          break;
        }
        tc_fence_after();
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % STAGES;
          const uint32_t ph = (it / STAGES) & 1;
          if (!mbar_wait(&full[s], ph, abort_flag, kTfWaitNs)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + s * STAGE_BYTES), sb = sa + A_BYTES;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint64_t ad = sw128_desc(sa + kk * 32, 16, 1024);
            // K-major B: 16 K-elements = 32 B along the row; MN-major B: 16 K rows =
            // two 8-row groups (2048 B), 64-column blocks one box apart
            const uint64_t bd = MN ? sw128_desc(sb + kk * 2048, BOX_MN_BYTES, 1024)
                                   : sw128_desc(sb + kk * 32, 16, 1024);
            mma_bf16(tmem + buf * BN, ad, bd, idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          }
          mma_commit(&empty[s]);
        }
        if (!ok) break;
        mma_commit(&accf[buf]);
      }
      if (!ok) {
        *abort_flag = 1;
        raise_error(a.st, FFH_ERR_TIMEOUT, 32);
      }
      mma_commit(drain);
      volatile int never = 0;
      mbar_wait(drain, 0, &never, kTfWaitNs);
    }
  } else if (warp >= 4) {
    const int wq = warp - 4;
    uint32_t cc = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < a.units && ok; u += gridDim.x, ++cc) {
      const int k = u / per_k, rem = u - k * per_k;
      const int rt = rem / a.CT, ct = rem - rt * a.CT;
      const int buf = cc & 1;
      if (!mbar_wait(&accf[buf], (cc >> 1) & 1, abort_flag, kTfWaitNs)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int r = rt * BM + wq * 32 + lane;
      __nv_bfloat16* vrow = a.V + ((int64_t)k * a.d_out + r) * a.ldv;
#pragma unroll 1
      for (int cb = 0; cb < BN / 32; ++cb) {
        float v[32];
        tmem_ld32(tmem + ((uint32_t)(wq * 32) << 16) + buf * BN + cb * 32, v);
        const int c0 = ct * BN + cb * 32;
        if (r < a.d_out) {
          if (c0 + 32 <= a.d_other) {
            uint4* dst = reinterpret_cast<uint4*>(vrow + c0);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              __nv_bfloat162 p0 = __floats2bfloat162_rn(v[8 * q + 0], v[8 * q + 1]);
              __nv_bfloat162 p1 = __floats2bfloat162_rn(v[8 * q + 2], v[8 * q + 3]);
              __nv_bfloat162 p2 = __floats2bfloat162_rn(v[8 * q + 4], v[8 * q + 5]);
              __nv_bfloat162 p3 = __floats2bfloat162_rn(v[8 * q + 6], v[8 * q + 7]);
              uint4 w;
              w.x = *reinterpret_cast<uint32_t*>(&p0);
              w.y = *reinterpret_cast<uint32_t*>(&p1);
              w.z = *reinterpret_cast<uint32_t*>(&p2);
              w.w = *reinterpret_cast<uint32_t*>(&p3);
              dst[q] = w;
            }
          } else {
            for (int jx = 0; jx < 32; ++jx)
              if (c0 + jx < a.d_other) vrow[c0 + jx] = __float2bfloat16_rn(v[jx]);
          }
        }
      }
      tc_fence_before();
      mbar_arrive(&acce[buf]);
    }
    if (!ok) {
      *abort_flag = 1;
      raise_error(a.st, FFH_ERR_TIMEOUT, 33);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// V rows (k, r) = (M Gop_k)[r][:] for the nk samples starting at Gb (bf16, sample k at
// Gb + k*m*n, row-major m x n).
//   b_update = true : Gop_k = G_k^T, d = n (M is n x n), output columns m
//   b_update = false: Gop_k = G_k,   d = m (M is m x m), output columns n
cudaError_t launch_transform_tc(const __nv_bfloat16* M, int64_t d, int64_t ldm,
                                const __nv_bfloat16* Gb, int64_t nk, int64_t m, int64_t n,
                                bool b_update, __nv_bfloat16* V, DevStatus* st, cudaStream_t s) {
  if (nk <= 0) return cudaSuccess;
  CUtensorMap mm, gm;
  if (!map2d_bf16(&mm, M, (uint64_t)d, (uint64_t)d, (uint64_t)ldm, 64, tf::BM))
    return cudaErrorInvalidValue;
  const int64_t d_other = b_update ? m : n;
  if (b_update) {
    // rows of all samples (k*m + c), K = j along n
    if (!map2d_bf16(&gm, Gb, (uint64_t)n, (uint64_t)(nk * m), (uint64_t)n, 64, tf::BN))
      return cudaErrorInvalidValue;
  } else {
    // rows (k*m + j), columns c along n, 64 x 64 boxes
    if (!map2d_bf16(&gm, Gb, (uint64_t)n, (uint64_t)(nk * m), (uint64_t)n, 64, tf::BK))
      return cudaErrorInvalidValue;
  }
  static PerDeviceOnce attr[2];
  {
    const void* fn = b_update ? (const void*)k_transform_tc<false> : (const void*)k_transform_tc<true>;
    cudaError_t e = smem_attr_once(fn, tf::SMEM_BYTES, attr[b_update ? 0 : 1]);
    if (e != cudaSuccess) return e;
  }
  TransformArgs a;
  a.V = V;
  a.ldv = d_other;
  a.d_out = (int)d;
  a.d_other = (int)d_other;
  a.d_in = (int)d;
  a.g_rows = (int)m;
  a.nk = (int)nk;
  a.RT = (int)((d + tf::BM - 1) / tf::BM);
  a.CT = (int)((d_other + tf::BN - 1) / tf::BN);
  a.units = (int)(nk * a.RT * a.CT);
  a.st = st;
  const int grid = std::min(a.units, num_sms());
  if (b_update)
    k_transform_tc<false><<<grid, tf::THREADS, tf::SMEM_BYTES, s>>>(mm, gm, a);
  else
    k_transform_tc<true><<<grid, tf::THREADS, tf::SMEM_BYTES, s>>>(mm, gm, a);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace ffh
