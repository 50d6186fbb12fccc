// Tensor-core Cholesky factor and triangular inverse of the d x d factors A, B.
//
// Blocked right-looking Cholesky with 128-wide panels (Section 2 notation: L lower,
// L L^T = F):
//   * k_chol_leaf  factors the 128 x 128 diagonal block in shared memory (one CTA) and,
//                  in the same column sweep, its inverse M11 = L11^-1 (each elimination
//                  step applied to the identity as well);
//   * the panel below, L21 = A21 M11^T, and the trailing update A22 -= L21 L21^T are
//     tcgen05 GEMMs (k_gemm_tc);
// then M = L^-1 by recursive doubling over the diagonal-block inverses:
//   [[L11, 0], [L21, L22]]^-1 = [[M11, 0], [-M22 (L21 M11), M22]].
//
// fp32 operands enter the bf16 tensor cores as a hi/lo split (x = hi + lo, both bf16):
// a b ~ hi_a hi_b + hi_a lo_b + lo_a hi_b, accumulated in fp32 (relative error of a
// product ~2^-16).  The split is laid out as [hi | lo] along K, so the three products
// are one GEMM over three K segments.
#include <cudaTypedefs.h>

#include <algorithm>

#include "ffh_internal.cuh"
#include "tc_ptx.cuh"

namespace ffh {

using namespace ptx;

static constexpr uint64_t kGemmWaitNs = 4000000000ull;

// Programmatic dependent launch: the kernels of the panel chain start (launch, CTA
// placement) while their predecessor in the stream is still running, and wait for it to
// finish, with its memory visible, before touching any data (griddepcontrol.wait).  A
// kernel lets its dependent start as soon as all of its own CTAs are resident.
__device__ __forceinline__ void pdl_enter() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
static cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

static PFN_cuTensorMapEncodeTiled_v12000 encode_fn_chol() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

static bool map_bf16_kmajor(CUtensorMap* m, const void* base, uint64_t k_extent, uint64_t rows,
                            uint64_t pitch_elems, uint32_t box_rows) {
  auto fn = encode_fn_chol();
  if (!fn) return false;
  cuuint64_t dims[2] = {k_extent, rows};
  cuuint64_t strides[1] = {pitch_elems * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ===========================================================================
// TN GEMM on tcgen05:  C[z] = alpha * A'[z] B'[z]^T + beta * C[z]
//   A'[z]: M x K' bf16 rows (K-major), B'[z]: N x K' bf16 rows (K-major); both are the
//   packed rows z*rows_pad .. of one 2-D buffer.  K' is a list of up to three 64-aligned
//   segments (x offsets per operand), each kseg wide.
//   C: fp32 row-major, element (r, c) of batch z at C + z*strideC + r*ldc + c.
// ===========================================================================
namespace gt {
constexpr int BM = 128, BN = 128, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2, B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + 256;
constexpr uint32_t TMEM_COLS = 128;
}  // namespace gt

struct GemmTcArgs {
  float* C;
  int64_t ldc, strideC;
  int M, N;                 // valid rows / cols of C per batch
  int a_rows_pad, b_rows_pad;  // packed rows per batch in the A' / B' buffers
  int nseg, kseg_blocks;    // segments, 64-blocks per segment
  int a_off[3], b_off[3];   // x offsets (elements) of the segments
  float alpha, beta;
  int lower_only;           // skip tiles strictly above the diagonal
  __nv_bfloat16* split_out; // optional: also write the bf16 hi/lo split of the result,
  int split_kpad;           //   row r of batch z at (z*M_pad + r) * 2*split_kpad
  int split_rows_pad;
  DevStatus* st;
};

__global__ void __launch_bounds__(256, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap bmap,
              const GemmTcArgs a) {
  using namespace gt;
  pdl_enter();
  const int tn = blockIdx.x, tm = blockIdx.y, z = blockIdx.z;
  const int row0 = tm * BM, col0 = tn * BN;
  if (a.lower_only && col0 > row0 + BM - 1) return;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;
  uint64_t* drain = accf + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* skip_flag = abort_flag + 1;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    *skip_flag = *reinterpret_cast<volatile int*>(&a.st->abort_all);
    *abort_flag = 0;
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accf, 1);
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
  const int nk = a.nseg * a.kseg_blocks;
  const int arow = z * a.a_rows_pad + row0, brow = z * a.b_rows_pad + col0;

  if (warp == 0 && lane == 0) {
    bool ok = true;
    int it = 0;
    for (; it < nk; ++it) {
      const int s = it % STAGES;
      const uint32_t ph = (it / STAGES) & 1;
      if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, kGemmWaitNs)) {
        ok = false;
        break;
      }
      const int seg = it / a.kseg_blocks, kb = it - seg * a.kseg_blocks;
      mbar_arrive_expect_tx(&full[s], STAGE_BYTES);
      uint8_t* sa = smem + s * STAGE_BYTES;
      tma_load_2d(sa, &amap, &full[s], a.a_off[seg] + kb * BK, arow);
      tma_load_2d(sa + A_BYTES, &bmap, &full[s], a.b_off[seg] + kb * BK, brow);
    }
    if (!ok) {
      *abort_flag = 1;
      raise_error(a.st, FFH_ERR_TIMEOUT, 21);
    }
    const int first = it > STAGES ? it - STAGES : 0;
    for (int j = first; j < it; ++j) {
      volatile int never = 0;
      mbar_wait(&full[j % STAGES], (j / STAGES) & 1, &never, kGemmWaitNs);
    }
  } else if (warp == 1 && lane == 0) {
    constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, false, false);
    bool ok = true;
    for (int it = 0; it < nk; ++it) {
      const int s = it % STAGES;
      const uint32_t ph = (it / STAGES) & 1;
      if (!mbar_wait(&full[s], ph, abort_flag, kGemmWaitNs)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + s * STAGE_BYTES), sb = sa + A_BYTES;
#pragma unroll
      for (int k = 0; k < BK / 16; ++k)
        mma_bf16(tmem, sw128_desc(sa + k * 32, 16, 1024), sw128_desc(sb + k * 32, 16, 1024),
                 idesc, (it > 0 || k > 0) ? 1u : 0u);
      mma_commit(&empty[s]);
    }
    if (ok) {
      mma_commit(accf);
    } else {
      *abort_flag = 1;
      raise_error(a.st, FFH_ERR_TIMEOUT, 22);
    }
    mma_commit(drain);
    volatile int never = 0;
    mbar_wait(drain, 0, &never, kGemmWaitNs);
  } else if (warp >= 4) {
    const int wq = warp - 4;
    if (mbar_wait(accf, 0, abort_flag, kGemmWaitNs)) {
      tc_fence_after();
      // every MMA has completed (accf), so the stage buffers are free: each warp
      // transposes its 32 x 32 chunks through shared memory and stores rows
      // contiguously across lanes.
      float* tb = reinterpret_cast<float*>(smem) + wq * 32 * 33;
      const int rbase = row0 + wq * 32;
#pragma unroll 1
      for (int cb = 0; cb < BN / 32; ++cb) {
        float v[32];
        tmem_ld32(tmem + ((uint32_t)(wq * 32) << 16) + cb * 32, v);
#pragma unroll
        for (int j = 0; j < 32; ++j) tb[lane * 33 + j] = v[j];
        __syncwarp();
        const int c = col0 + cb * 32 + lane;
        float* cbase = a.C + (int64_t)z * a.strideC + (int64_t)rbase * a.ldc + c;
        // all loads of C first (independent, in flight together), then the stores
        float prev[32];
        if (a.beta != 0.f) {
#pragma unroll
          for (int rr = 0; rr < 32; ++rr)
            prev[rr] = (rbase + rr < a.M && c < a.N) ? cbase[(int64_t)rr * a.ldc] : 0.f;
        }
#pragma unroll
        for (int rr = 0; rr < 32; ++rr) {
          const int r = rbase + rr;
          if (r < a.M && c < a.N) {
            const float o = a.alpha * tb[rr * 33 + lane];
            const float res = a.beta == 0.f ? o : fmaf(a.beta, prev[rr], o);
            cbase[(int64_t)rr * a.ldc] = res;
            if (a.split_out) {
              __nv_bfloat16* srow =
                  a.split_out + ((int64_t)z * a.split_rows_pad + r) * 2 * a.split_kpad;
              const __nv_bfloat16 hi = __float2bfloat16_rn(res);
              srow[c] = hi;
              srow[a.split_kpad + c] = __float2bfloat16_rn(res - __bfloat162float(hi));
            }
          }
        }
        __syncwarp();
      }
      tc_fence_before();
    } else {
      *abort_flag = 1;
      raise_error(a.st, FFH_ERR_TIMEOUT, 23);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// A bf16 hi/lo split buffer: rows x [hi (kpad) | lo (kpad)], pitch 2*kpad, kpad = 64-aligned.
struct Split {
  __nv_bfloat16* p;
  int rows_pad;   // packed rows per batch (>= valid rows; rows beyond are masked outputs)
  int kpad;       // 64-aligned K extent of one half
  int batch;
};

static cudaError_t gemm_tc(const Split& A, const Split& B, int nseg, const int a_seg[3],
                           const int b_seg[3], int kseg, float* C, int64_t ldc, int64_t strideC,
                           int M, int N, float alpha, float beta, bool lower_only, int batch,
                           DevStatus* st, cudaStream_t s, const Split* out_split = nullptr) {
  if (M <= 0 || N <= 0 || batch <= 0) return cudaSuccess;
  CUtensorMap am, bm;
  if (!map_bf16_kmajor(&am, A.p, (uint64_t)2 * A.kpad, (uint64_t)A.rows_pad * A.batch,
                       (uint64_t)2 * A.kpad, gt::BM))
    return cudaErrorInvalidValue;
  if (!map_bf16_kmajor(&bm, B.p, (uint64_t)2 * B.kpad, (uint64_t)B.rows_pad * B.batch,
                       (uint64_t)2 * B.kpad, gt::BN))
    return cudaErrorInvalidValue;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(k_gemm_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         gt::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  GemmTcArgs g{};
  g.C = C;
  g.ldc = ldc;
  g.strideC = strideC;
  g.M = M;
  g.N = N;
  g.a_rows_pad = A.rows_pad;
  g.b_rows_pad = B.rows_pad;
  g.nseg = nseg;
  g.kseg_blocks = (kseg + 63) / 64;
  for (int i = 0; i < 3; ++i) {
    g.a_off[i] = a_seg[i];
    g.b_off[i] = b_seg[i];
  }
  g.alpha = alpha;
  g.beta = beta;
  g.lower_only = lower_only ? 1 : 0;
  g.split_out = out_split ? out_split->p : nullptr;
  g.split_kpad = out_split ? out_split->kpad : 0;
  g.split_rows_pad = out_split ? out_split->rows_pad : 0;
  g.st = st;
  dim3 grid((N + gt::BN - 1) / gt::BN, (M + gt::BM - 1) / gt::BM, batch);
  cudaError_t e = launch_pdl(k_gemm_tc, grid, dim3(256), gt::SMEM_BYTES, s, am, bm, g);
  note_launches(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// ---------------------------------------------------------------------------
// fp32 -> bf16 hi/lo split, optionally transposed, batched:
//   batch z, row r < rows, col c < cols of the source view
//     src[z*src_stride + r*lds + c]          (trans = 0)
//     src[z*src_stride + c*lds + r]          (trans = 1: output row r = source column r)
//   dst[(z*rows_pad + r)*2kpad + c] = hi, [... + kpad + c] = lo; zero elsewhere up to
//   rows_pad x 2kpad.
// ---------------------------------------------------------------------------
__global__ void k_split_hilo(const float* __restrict__ src, int64_t lds, int64_t src_stride,
                             int rows, int cols, int trans, __nv_bfloat16* __restrict__ dst,
                             int rows_pad, int kpad, int batch) {
  pdl_enter();
  const int64_t per = (int64_t)rows_pad * kpad;
  const int64_t total = per * batch;
  for (int64_t idx = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (int64_t)gridDim.x * blockDim.x) {
    const int z = (int)(idx / per);
    const int64_t rem = idx - (int64_t)z * per;
    const int r = (int)(rem / kpad), c = (int)(rem - (int64_t)r * kpad);
    float x = 0.f;
    if (r < rows && c < cols) {
      const float* sz = src + (int64_t)z * src_stride;
      x = trans ? sz[(int64_t)c * lds + r] : sz[(int64_t)r * lds + c];
    }
    const __nv_bfloat16 hi = __float2bfloat16_rn(x);
    const __nv_bfloat16 lo = __float2bfloat16_rn(x - __bfloat162float(hi));
    __nv_bfloat16* drow = dst + ((int64_t)z * rows_pad + r) * (2 * (int64_t)kpad);
    drow[c] = hi;
    drow[kpad + c] = lo;
  }
}

static cudaError_t split(const float* src, int64_t lds, int64_t src_stride, int rows, int cols,
                         bool trans, const Split& d, cudaStream_t s) {
  const int64_t total = (int64_t)d.rows_pad * d.kpad * d.batch;
  if (total == 0) return cudaSuccess;
  const int64_t blocks = std::min<int64_t>((total + 255) / 256, (int64_t)num_sms() * 16);
  cudaError_t e = launch_pdl(k_split_hilo, dim3((unsigned)blocks), dim3(256), 0, s, src, lds,
                             src_stride, rows, cols, trans ? 1 : 0, d.p, d.rows_pad, d.kpad,
                             d.batch);
  note_launches(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// ---------------------------------------------------------------------------
// 128 x 128 diagonal block: Cholesky factor L11 and inverse M11 = L11^-1, one CTA of
// 512 threads (16 warps), blocked by 32 (sub-panels q = 0..3, rows/cols Q = [32q, 32q+32)).
//   A(q)  warp 0 factors the 32 x 32 diagonal block D_q and inverts it in registers:
//         lane i holds row i of D_q and column i of its inverse; pivot j is broadcast
//         by shuffle, and the remaining columns shift down one register per pivot so
//         every register index is static.  Writes L_qq, Mi_q = L_qq^-1 and
//         Mt[x][k] = Mi_q[k][x].
//   B(q)  all warps: the rows below, L[r][Q] = A[r][Q] Mi_q^T (4 x 4 register blocks),
//         also stored transposed, Pt[k][r] = L[r][32q+k].
//   C(q)  warps 0-1 apply the rank-32 update of sub-panel q to D_{q+1} and warp 0 goes
//         on to A(q+1), while 11 other warps (not 4, 8, 12, which share warp 0's
//         scheduler partition) update the rest of the trailing lower triangle
//         and form row block q of the inverse by block forward substitution,
//         M[Q][0:32q] = -Mi_q T_q, and the product T_{q+1} = L[Q+1][0:32q+32] M[..][..]
//         of the next row block (only -Mi_3 T_3 is left after the last sub-panel).
// Pt and Mt are double-buffered by the parity of q, so A(q+1) never writes what C(q)
// reads.  The pivot product gives log|F11| = sum_j log(pivot_j).
// Outputs: L11 and M11 (fp32) and the bf16 hi/lo split of M11 ([hi | lo] rows, pitch
// 256), the B operand of the panel GEMM.
// ---------------------------------------------------------------------------
constexpr int LB = 128;
constexpr int LP = LB + 1;   // pitch of the row-major 128 x 128 blocks (conflict-free columns)
constexpr int PTP = LB + 4;  // pitch of Pt (float4 rows)
constexpr int MP = LB + 4;   // pitch of M11 (float4 rows)
constexpr int MTP = 36;      // pitch of Mt
constexpr int TP = 100;      // pitch of the 32 x 96 scratch T
constexpr int LB_SMEM =
    (LB * LP + LB * MP + 2 * 32 * PTP + 2 * 32 * MTP + 32 * TP + LB + 64) * 4 + 64;
constexpr int LEAF_THREADS = 512;

// A(q): factor and invert the diagonal block (warp 0 only); the pivots go to pivs[c0..].
// The column of l values of pivot j reaches the other lanes through a shared buffer
// written rotated (slot (lane - j - 1) mod 32 holds lane lane's value), so the 31 values
// l_{j+1..j+31, j} are eight broadcast float4 loads; the buffer alternates by the parity of
// j, so one warp barrier per pivot suffices.  Not inlined: one copy serves the four
// sub-panels (measured faster than the inlined copies).
__device__ __noinline__ void leaf_diag(float* Ls, float* Ms, float* Mt, float* lbuf,
                                          float* pivs, int c0, int64_t o, DevStatus* st,
                                          bool& bad) {
  const int lane = threadIdx.x & 31;
  constexpr unsigned FULL = 0xffffffffu;
  float a[32], mc[32];
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    a[k] = (k <= lane) ? Ls[(c0 + lane) * LP + c0 + k] : 0.f;
    mc[k] = (k == lane) ? 1.f : 0.f;
  }
#pragma unroll 1
  for (int j = 0; j < 32; ++j) {
    // registers k = 0..31 hold columns j+k of row `lane` (of D) and rows j+k of column
    // `lane` (of the inverse)
    float piv = __shfl_sync(FULL, a[0], j);
    if (!(piv > 0.f) || !isfinite(piv)) {  // warp-uniform (broadcast value)
      if (lane == 0 && !bad) raise_error(st, FFH_ERR_NOT_SPD, (int)(o + c0 + j));
      bad = true;
      piv = 1.f;
    }
    // 1/sqrt to within 2 ulp; far below the fp32 accumulation error of the updates
    const float r = rsqrtf(piv);
    const float l = a[0] * r;   // lane > j: l_{lane,j}; lane j: sqrt(pivot)
    const float m = mc[0] * r;  // Mi[j][lane] (exactly 0 for lane > j)
    float* lb = lbuf + (j & 1) * 32;
    lb[(lane - j - 1) & 31] = l;
    if (lane == 0) pivs[c0 + j] = piv;
    Ls[(c0 + lane) * LP + c0 + j] = lane >= j ? l : 0.f;
    Ms[(c0 + j) * MP + c0 + lane] = m;
    Mt[lane * MTP + j] = m;
    __syncwarp();
    float lk[32];
#pragma unroll
    for (int k4 = 0; k4 < 8; ++k4) {
      const float4 v = *reinterpret_cast<const float4*>(lb + 4 * k4);
      lk[4 * k4] = v.x;
      lk[4 * k4 + 1] = v.y;
      lk[4 * k4 + 2] = v.z;
      lk[4 * k4 + 3] = v.w;
    }
#pragma unroll
    for (int k = 1; k < 32; ++k) {
      // lk[k-1] = l_{j+k, j}; for j + k > 31 the value is unused (shifted past the block)
      a[k - 1] = fmaf(-l, lk[k - 1], a[k]);
      mc[k - 1] = fmaf(-lk[k - 1], m, mc[k]);
    }
    a[31] = 0.f;
    mc[31] = 0.f;
  }
}

// Rank-32 update of one 4 x 4 block of the trailing lower triangle from the transposed
// sub-panel: A[r][c] -= sum_k Pt[k][r] Pt[k][c].
__device__ __forceinline__ void leaf_trail_block(float* Ls, const float* Pt, int r0, int cc0) {
  float acc[4][4] = {};
#pragma unroll 8
  for (int k = 0; k < 32; ++k) {
    const float4 av = *reinterpret_cast<const float4*>(Pt + k * PTP + r0);
    const float4 bv = *reinterpret_cast<const float4*>(Pt + k * PTP + cc0);
    const float ar[4] = {av.x, av.y, av.z, av.w}, br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int jx = 0; jx < 4; ++jx) acc[i][jx] = fmaf(ar[i], br[jx], acc[i][jx]);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int jx = 0; jx < 4; ++jx)
      if (cc0 + jx <= r0 + i) Ls[(r0 + i) * LP + cc0 + jx] -= acc[i][jx];
}

// Row block Q = [c0, c0 + 32) (c0 >= 32) of the inverse, left of the diagonal block, in
// two products: T = L[Q][0:c0] M[0:c0][0:c0] (needs the rows of M above Q), then
// M[Q][0:c0] = -Mi_Q T (needs the diagonal block's inverse Mi_Q).  Threads t = 0..nt-1.
__device__ __forceinline__ void leaf_inverse_T(const float* Ls, const float* Ms, float* T, int c0,
                                               int t, int nt) {
  const int nbx = c0 / 4;  // 4-wide column blocks of [0, c0)
  // 2 rows x 4 columns per thread
  for (int blk = t; blk < 16 * nbx; blk += nt) {
    const int i0 = (blk / nbx) * 2, x0 = (blk % nbx) * 4;
    float acc[2][4] = {};
    // M lower triangular: M[k][x] = 0 for k < x, so k starts at x0
    for (int k = x0; k < c0; ++k) {
      float av[2];
#pragma unroll
      for (int i = 0; i < 2; ++i) av[i] = Ls[(c0 + i0 + i) * LP + k];
      const float4 bv = *reinterpret_cast<const float4*>(Ms + k * MP + x0);
      const float br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
      for (int i = 0; i < 2; ++i)
#pragma unroll
        for (int jx = 0; jx < 4; ++jx) acc[i][jx] = fmaf(av[i], br[jx], acc[i][jx]);
    }
#pragma unroll
    for (int i = 0; i < 2; ++i)
      *reinterpret_cast<float4*>(T + (i0 + i) * TP + x0) =
          make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
  }
}

__device__ __forceinline__ void leaf_inverse_apply(float* Ms, const float* T, int c0, int t,
                                                   int nt) {
  const int nbx = c0 / 4;
  // 2 rows x 4 columns per thread
  for (int blk = t; blk < 16 * nbx; blk += nt) {
    const int i0 = (blk / nbx) * 2, x0 = (blk % nbx) * 4;
    float acc[2][4] = {};
    // Mi lower triangular: row i needs j <= i < i0 + 2
    for (int j = 0; j < i0 + 2; ++j) {
      float av[2];
#pragma unroll
      for (int i = 0; i < 2; ++i) av[i] = Ms[(c0 + i0 + i) * MP + c0 + j];
      const float4 bv = *reinterpret_cast<const float4*>(T + j * TP + x0);
      const float br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
      for (int i = 0; i < 2; ++i)
#pragma unroll
        for (int jx = 0; jx < 4; ++jx) acc[i][jx] = fmaf(av[i], br[jx], acc[i][jx]);
    }
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int jx = 0; jx < 4; ++jx) Ms[(c0 + i0 + i) * MP + x0 + jx] = -acc[i][jx];
  }
}

__global__ void __launch_bounds__(LEAF_THREADS, 1) k_chol_leaf(float* W, int64_t ldw, int64_t d,
                                                               int64_t o, float* L, int64_t ldl,
                                                               float* Minv, int64_t ldm,
                                                               __nv_bfloat16* m11_split,
                                                               DevStatus* st, int fault) {
  extern __shared__ float sh[];
  float* Ls = sh;                      // [LB][LP]  working block -> L11
  float* Ms = Ls + LB * LP;            // [LB][MP]  M11
  float* Ptb = Ms + LB * MP;           // [2][32][PTP] transposed sub-panels
  float* Mtb = Ptb + 2 * 32 * PTP;     // [2][32][MTP] transposed diagonal-block inverses
  float* T = Mtb + 2 * 32 * MTP;       // [32][TP]
  float* pivs = T + 32 * TP;           // [LB] pivots
  float* lbuf = pivs + LB;             // [2][32] pivot-column broadcast (warp 0)
  pdl_enter();
  const int b = (int)((d - o) < LB ? (d - o) : LB);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  for (int idx = tid; idx < LB * LB / 4; idx += LEAF_THREADS) {
    const int i = idx >> 5, j4 = (idx & 31) * 4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i < b) {
      const float* src = W + (o + i) * ldw + o + j4;
      if (j4 + 3 < b && (((uintptr_t)src) & 15) == 0) {
        v = *reinterpret_cast<const float4*>(src);
      } else {
        if (j4 + 0 < b) v.x = src[0];
        if (j4 + 1 < b) v.y = src[1];
        if (j4 + 2 < b) v.z = src[2];
        if (j4 + 3 < b) v.w = src[3];
      }
    }
    const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int j = j4 + e;
      float x = (j <= i) ? vv[e] : 0.f;
      if (i >= b || j >= b) x = (i == j) ? 1.f : 0.f;  // identity padding
      Ls[i * LP + j] = x;
      Ms[i * MP + j] = 0.f;
    }
  }
  __syncthreads();
  if (tid == 0 && fault == FFH_FAULT_BAD_PIVOT && o == 0) Ls[0] = __int_as_float(0x7fc00000);
  __syncthreads();
  bool bad = false;
  if (warp == 0) leaf_diag(Ls, Ms, Mtb, lbuf, pivs, 0, o, st, bad);
  __syncthreads();
#pragma unroll 1
  for (int q = 0; q < 4; ++q) {
    const int c0 = 32 * q;
    float* Pt = Ptb + (q & 1) * 32 * PTP;
    const float* Mt = Mtb + (q & 1) * 32 * MTP;
    // B(q): rows r in [c0 + 32, 128) of the sub-panel, L[r][c0 + k] = sum_x A[r][c0 + x] Mi[k][x].
    // At most one 4 x 4 block per thread; results are held across a barrier because the
    // blocks of a row read the A entries that other blocks of the row overwrite.
    const int R = LB - c0 - 32;
    const bool has = tid < (R / 4) * 8;
    const int r0 = c0 + 32 + (tid >> 3) * 4, k0 = (tid & 7) * 4;
    float acc[4][4] = {};
    if (has) {
      for (int x = 0; x < k0 + 4; ++x) {  // Mi[k][x] = 0 for x > k
        float av[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) av[i] = Ls[(r0 + i) * LP + c0 + x];
        const float4 bv = *reinterpret_cast<const float4*>(Mt + x * MTP + k0);
        const float br[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int jx = 0; jx < 4; ++jx) acc[i][jx] = fmaf(av[i], br[jx], acc[i][jx]);
      }
    }
    __syncthreads();
    if (has) {
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int jx = 0; jx < 4; ++jx) Ls[(r0 + i) * LP + c0 + k0 + jx] = acc[i][jx];
#pragma unroll
      for (int jx = 0; jx < 4; ++jx)
        *reinterpret_cast<float4*>(Pt + (k0 + jx) * PTP + r0) =
            make_float4(acc[0][jx], acc[1][jx], acc[2][jx], acc[3][jx]);
    }
    __syncthreads();
    if (q < 3) {
      const int nb = R / 4;  // 4-row blocks of the trailing matrix [c0 + 32, 128)
      if (warp < 2) {
        // D_{q+1} first (4-blocks bi, bj < 8), then warp 0 factors it
        const int bi = tid >> 3, bj = tid & 7;
        if (bj <= bi) leaf_trail_block(Ls, Pt, c0 + 32 + 4 * bi, c0 + 32 + 4 * bj);
        asm volatile("bar.sync 1, 64;" ::: "memory");
        if (warp == 0)
          leaf_diag(Ls, Ms, Mtb + ((q + 1) & 1) * 32 * MTP, lbuf, pivs, c0 + 32, o, st, bad);
      } else if (warp & 3) {
        // warps 2, 3, 5-7, 9-11, 13-15: warps 4, 8 and 12 stay idle so that warp 0's
        // pivot chain has its scheduler partition to itself
        constexpr int NT = 11 * 32;
        const int t = (warp - 2 - (warp >> 2)) * 32 + (tid & 31);
        for (int blk = t; blk < nb * nb; blk += NT) {
          const int bi = blk / nb, bj = blk - (blk / nb) * nb;
          if (bi < 8 || bj > bi) continue;
          leaf_trail_block(Ls, Pt, c0 + 32 + 4 * bi, c0 + 32 + 4 * bj);
        }
        // row block q of the inverse (T_q from the previous sub-panel), then T_{q+1}
        if (q >= 1) {
          leaf_inverse_apply(Ms, T, c0, t, NT);
          asm volatile("bar.sync 2, 352;" ::: "memory");
        }
        leaf_inverse_T(Ls, Ms, T, c0 + 32, t, NT);
      }
    } else {
      leaf_inverse_apply(Ms, T, c0, tid, LEAF_THREADS);
    }
    __syncthreads();
  }
  // write-out, four consecutive columns per thread
  const bool vec_ok = ((ldl | ldm) & 3) == 0 && (o & 3) == 0 &&
                      ((reinterpret_cast<uintptr_t>(L) | reinterpret_cast<uintptr_t>(Minv)) & 15) == 0;
  for (int idx = tid; idx < LB * LB / 4; idx += LEAF_THREADS) {
    const int i = idx >> 5, j0 = (idx & 31) * 4;
    float lv[4], mv[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int j = j0 + e;
      lv[e] = (j <= i) ? Ls[i * LP + j] : 0.f;
      mv[e] = (j <= i && i < b && j < b) ? Ms[i * MP + j] : 0.f;
    }
    if (i < b) {
      if (vec_ok && j0 + 3 < b) {
        *reinterpret_cast<float4*>(L + (o + i) * ldl + o + j0) = make_float4(lv[0], lv[1], lv[2], lv[3]);
        *reinterpret_cast<float4*>(Minv + (o + i) * ldm + o + j0) =
            make_float4(mv[0], mv[1], mv[2], mv[3]);
      } else {
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (j0 + e < b) {
            L[(o + i) * ldl + o + j0 + e] = lv[e];
            Minv[(o + i) * ldm + o + j0 + e] = mv[e];
          }
      }
    }
    if (m11_split) {
      __nv_bfloat16 hi[4], lo[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        hi[e] = __float2bfloat16_rn(mv[e]);
        lo[e] = __float2bfloat16_rn(mv[e] - __bfloat162float(hi[e]));
      }
      *reinterpret_cast<uint2*>(m11_split + i * 2 * LB + j0) = *reinterpret_cast<uint2*>(hi);
      *reinterpret_cast<uint2*>(m11_split + i * 2 * LB + LB + j0) = *reinterpret_cast<uint2*>(lo);
    }
  }
  if (warp == 0) {
    // log|F11| = sum_j log(pivot_j), off the pivot chain
    float lg = 0.f;
    for (int i = lane; i < LB; i += 32) lg += logf(pivs[i]);
    for (int off = 16; off > 0; off >>= 1) lg += __shfl_down_sync(0xffffffffu, lg, off);
    if (lane == 0) atomicAdd(&st->logdet, (double)lg);
  }
}

size_t cholesky_tc_work_bytes(int64_t d) {
  const int64_t kmax = (d + 63) / 64 * 64;
  const int64_t rows = (d + 127) / 128 * 128 + 128;
  // W copy, T scratch, five split buffers (each <= rows x 2*kmax bf16), each region and the
  // base rounded up to 256 bytes
  return (size_t)d * d * 4 + (size_t)d * d * 4 + 5 * (size_t)rows * 2 * kmax * 2 + 8 * 256 + 4096;
}

cudaError_t chol_streams_init(CholStreams* cs) {
  int least = 0, greatest = 0;
  cudaError_t e = cudaDeviceGetStreamPriorityRange(&least, &greatest);
  if (e != cudaSuccess) return e;
  if ((e = cudaStreamCreateWithPriority(&cs->crit, cudaStreamNonBlocking, greatest)) != cudaSuccess)
    return e;
  if ((e = cudaStreamCreateWithPriority(&cs->side, cudaStreamNonBlocking, least)) != cudaSuccess)
    return e;
  for (cudaEvent_t& ev : cs->ev)
    if ((e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming)) != cudaSuccess) return e;
  return cudaSuccess;
}

void chol_streams_destroy(CholStreams* cs) {
  if (cs->crit) cudaStreamSynchronize(cs->crit);
  if (cs->side) cudaStreamSynchronize(cs->side);
  for (cudaEvent_t& ev : cs->ev)
    if (ev) cudaEventDestroy(ev), ev = nullptr;
  if (cs->crit) cudaStreamDestroy(cs->crit), cs->crit = nullptr;
  if (cs->side) cudaStreamDestroy(cs->side), cs->side = nullptr;
}

static cudaError_t cholesky_tc_body(const float* F, int64_t d, int64_t ldf, float* L, float* Linv,
                                    void* work, DevStatus* st, int fault, cudaStream_t s,
                                    CholStreams* cs);

// L (lower), Linv = L^-1 (lower); st->logdet += log|F|.  F is read, not modified.
// Look-ahead (cs): panel p's trailing update is split into the next column block (on the
// critical stream, needed by panel p+1) and the columns beyond it (on the side stream,
// overlapping panel p+1's diagonal block and panel solve).  The update of a column block
// by panel p-1 (side) finishes before panel p updates the same block (critical), and the
// panel GEMM output buffer alternates between two splits so that the side stream's reads
// of panel p's split are not overwritten by panel p+1.
cudaError_t launch_cholesky_tc(const float* F, int64_t d, int64_t ldf, float* L, float* Linv,
                               void* work, DevStatus* st, int fault, cudaStream_t s_user,
                               CholStreams* cs) {
  cudaError_t e;
  cudaStream_t s = s_user;
  if (cs) {
    if ((e = cudaEventRecord(cs->ev[0], s_user)) != cudaSuccess) return e;
    if ((e = cudaStreamWaitEvent(cs->crit, cs->ev[0], 0)) != cudaSuccess) return e;
    if ((e = cudaStreamWaitEvent(cs->side, cs->ev[0], 0)) != cudaSuccess) return e;
    s = cs->crit;
  }
  e = cholesky_tc_body(F, d, ldf, L, Linv, work, st, fault, s, cs);
  if (cs) {
    // join: everything on both streams completes before later work on the user stream
    cudaEventRecord(cs->ev[2], cs->side);
    cudaStreamWaitEvent(cs->crit, cs->ev[2], 0);
    cudaEventRecord(cs->ev[4], cs->crit);
    cudaError_t e2 = cudaStreamWaitEvent(s_user, cs->ev[4], 0);
    if (e == cudaSuccess) e = e2;
  }
  return e;
}

static cudaError_t cholesky_tc_body(const float* F, int64_t d, int64_t ldf, float* L, float* Linv,
                                    void* work, DevStatus* st, int fault, cudaStream_t s,
                                    CholStreams* cs) {
  cudaError_t e;
  const int64_t kmax = (d + 63) / 64 * 64;
  const int64_t rows_cap = (d + 127) / 128 * 128 + 128;
  // every region starts on a 256-byte boundary (the split buffers are TMA sources, which
  // need 16-byte aligned bases; d x d fp32 regions are not multiples of 16 bytes for odd d)
  auto up = [](size_t b) { return (b + 255) / 256 * 256; };
  char* wp = static_cast<char*>(work);
  wp = reinterpret_cast<char*>(up(reinterpret_cast<uintptr_t>(wp)));
  float* W = reinterpret_cast<float*>(wp);
  wp += up((size_t)d * d * 4);
  float* T = reinterpret_cast<float*>(wp);
  wp += up((size_t)d * d * 4);
  __nv_bfloat16* sb[5];
  for (int i = 0; i < 5; ++i) {
    sb[i] = reinterpret_cast<__nv_bfloat16*>(wp);
    wp += up((size_t)rows_cap * 2 * kmax * 2);
  }
  static bool attr = false;
  if (!attr) {
    if ((e = cudaFuncSetAttribute(k_chol_leaf, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  LB_SMEM)) != cudaSuccess)
      return e;
    attr = true;
  }
  if ((e = cudaMemcpy2DAsync(W, d * 4, F, ldf * 4, d * 4, d, cudaMemcpyDeviceToDevice, s)) !=
      cudaSuccess)
    return e;
  if ((e = cudaMemsetAsync(L, 0, (size_t)d * d * 4, s)) != cudaSuccess) return e;
  if (Linv && (e = cudaMemsetAsync(Linv, 0, (size_t)d * d * 4, s)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(&st->logdet, 0, sizeof(double), s)) != cudaSuccess) return e;
  float* Mdiag = Linv ? Linv : T;  // the diagonal-block inverses (T is free until the inverse)
  const int np = (int)((d + LB - 1) / LB);
  for (int p = 0; p < np; ++p) {
    const int64_t o = (int64_t)p * LB;
    if ((e = launch_pdl(k_chol_leaf, dim3(1), dim3(LEAF_THREADS), LB_SMEM, s, W, d, d, o, L, d,
                        Mdiag, d, sb[1], st, fault)) != cudaSuccess)
      return e;
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const int rows = (int)(d - o - LB);
    if (rows <= 0) continue;
    // L21 = A21 * M11^T : A' = split(A21) (rows x 128), B' = split(M11) (128 x 128).  The
    // A21 split sits 128 rows into sb[0]: with look-ahead the previous panel's update of
    // this column block writes it from its epilogue (rows of the diagonal block first).
    Split a21{sb[0] + (size_t)LB * 2 * 128, (int)((rows + 127) / 128 * 128), 128, 1};
    Split m11{sb[1], 128, 128, 1};
    if ((!cs || p == 0) &&
        (e = split(W + (o + LB) * d + o, d, 0, rows, LB, false, a21, s)) != cudaSuccess)
      return e;
    const int aseg[3] = {0, 0, 128}, bseg[3] = {0, 128, 0};
    // the epilogue also writes the split of L21 for the trailing update
    const int rows_pad = (rows + 127) / 128 * 128;
    Split l21{sb[cs ? 2 + 2 * (p & 1) : 2], rows_pad, 128, 1};
    if ((e = gemm_tc(a21, m11, 3, aseg, bseg, 128, L + (o + LB) * d + o, d, 0, rows, LB, 1.f,
                     0.f, false, 1, st, s, &l21)) != cudaSuccess)
      return e;
    if (!cs) {
      // A22 -= L21 L21^T (lower tiles)
      if ((e = gemm_tc(l21, l21, 3, aseg, bseg, 128, W + (o + LB) * d + (o + LB), d, 0, rows,
                       rows, -1.f, 1.f, true, 1, st, s)) != cudaSuccess)
        return e;
      continue;
    }
    // side: columns beyond the next block, A22[128:, 128:] -= L21[128:] L21[128:]^T
    if ((e = cudaEventRecord(cs->ev[1], s)) != cudaSuccess) return e;
    if ((e = cudaStreamWaitEvent(cs->side, cs->ev[1], 0)) != cudaSuccess) return e;
    if (rows > LB) {
      Split rest{l21.p + (size_t)LB * 2 * l21.kpad, rows_pad - LB, 128, 1};
      if ((e = gemm_tc(rest, rest, 3, aseg, bseg, 128, W + (o + 2 * LB) * d + (o + 2 * LB), d, 0,
                       rows - LB, rows - LB, -1.f, 1.f, true, 1, st, cs->side)) != cudaSuccess)
        return e;
    }
    if ((e = cudaEventRecord(cs->ev[2 + (p & 1)], cs->side)) != cudaSuccess) return e;
    // critical: the next column block, A22[:, :128] -= L21 L21[:128]^T, after the side
    // stream's update of the same block by the previous panel
    if (p > 0 && (e = cudaStreamWaitEvent(s, cs->ev[2 + ((p - 1) & 1)], 0)) != cudaSuccess)
      return e;
    Split head{l21.p, LB, 128, 1};
    Split next_a21{sb[0], rows_pad + LB, 128, 1};  // the next panel's A21 split (see above)
    if ((e = gemm_tc(l21, head, 3, aseg, bseg, 128, W + (o + LB) * d + (o + LB), d, 0, rows,
                     rows < LB ? rows : LB, -1.f, 1.f, true, 1, st, s,
                     rows > LB ? &next_a21 : nullptr)) != cudaSuccess)
      return e;
  }
  if (cs) {
    // the side stream's last updates precede the inverse
    if ((e = cudaEventRecord(cs->ev[2 + (np & 1)], cs->side)) != cudaSuccess) return e;
    if ((e = cudaStreamWaitEvent(s, cs->ev[2 + (np & 1)], 0)) != cudaSuccess) return e;
  }
  if (!Linv) return cudaSuccess;
  // inverse by recursive doubling over block size b = 128, 256, ...
  for (int64_t b = LB; b < d; b *= 2) {
    const int64_t full_pairs = d / (2 * b);
    const int64_t o_last = full_pairs * 2 * b;
    const int64_t rows_last = d - o_last - b;
    for (int part = 0; part < 2; ++part) {
      const int batch = (int)(part == 0 ? full_pairs : (rows_last > 0 ? 1 : 0));
      if (batch == 0) continue;
      const int64_t o = part == 0 ? 0 : o_last;
      const int rows = (int)(part == 0 ? b : rows_last);
      const int64_t zs = 2 * b * d + 2 * b;  // source stride between pairs
      const int kb = (int)((b + 63) / 64 * 64);
      const int kr = (rows + 63) / 64 * 64;
      const int rp = (rows + 127) / 128 * 128;
      const int bp = (int)((b + 127) / 128 * 128);
      // T_z = L21_z M11_z : A' = split(L21) (rows x b), B' = split(M11^T) (b x b)
      Split l21{sb[0], rp, kb, batch};
      Split m11t{sb[1], bp, kb, batch};
      if ((e = split(L + (o + b) * d + o, d, zs, rows, (int)b, false, l21, s)) != cudaSuccess)
        return e;
      if ((e = split(Linv + o * d + o, d, zs, (int)b, (int)b, true, m11t, s)) != cudaSuccess)
        return e;
      const int as1[3] = {0, 0, kb}, bs1[3] = {0, kb, 0};
      if ((e = gemm_tc(l21, m11t, 3, as1, bs1, (int)b, T, b, (int64_t)rp * b, rows, (int)b, 1.f,
                       0.f, false, batch, st, s)) != cudaSuccess)
        return e;
      // M21_z = -M22_z T_z : A' = split(M22) (rows x rows), B' = split(T^T) (b x rows)
      Split m22{sb[2], rp, kr, batch};
      Split tt{sb[3], bp, kr, batch};
      if ((e = split(Linv + (o + b) * d + (o + b), d, zs, rows, rows, false, m22, s)) !=
          cudaSuccess)
        return e;
      // B'[c][k] = T[k][c]: b output rows, `rows` output columns
      if ((e = split(T, b, (int64_t)rp * b, (int)b, rows, true, tt, s)) != cudaSuccess) return e;
      const int as2[3] = {0, 0, kr}, bs2[3] = {0, kr, 0};
      if ((e = gemm_tc(m22, tt, 3, as2, bs2, rows, Linv + (o + b) * d + o, d, zs, rows, (int)b,
                       -1.f, 0.f, false, batch, st, s)) != cudaSuccess)
        return e;
    }
  }
  return cudaSuccess;
}

}  // namespace ffh
