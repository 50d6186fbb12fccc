// Tensor-core Cholesky factor and triangular inverse of the d x d factors A, B.
//
// Blocked right-looking Cholesky with 128-wide panels (Section 2 notation: L lower,
// L L^T = F):
//   * k_chol_leaf  factors the 128 x 128 diagonal block in shared memory (one CTA) and,
//                  in the same column sweep, its inverse M11 = L11^-1 (each elimination
//                  step applied to the identity as well);
//   * the panel below, L21 = A21 M11^T, and the trailing update of the next column
//     block are tcgen05 GEMMs (k_gemm_tc); the trailing update A22 -= L21 L21^T of the
//     columns beyond it is a persistent tcgen05 kernel on a side stream (k_syrk_tc);
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
// Epilogue (when C's rows and batches start on 16-byte boundaries): all eight warps take
// a quarter of the tile's rows (their TMEM lane quarter) and half of its columns; each
// 32 x 32 block goes TMEM -> registers -> 128-byte-swizzled shared memory -> TMA tensor
// store, and beta C arrives the same way, loaded by TMA while the MMAs run.  The optional
// bf16 hi/lo split of the result is staged and stored the same way.  Other C layouts
// take a per-element epilogue (four warps, rows through a shared transpose).
// ===========================================================================
namespace gt {
constexpr int BM = 128, BN = 128, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2, B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int BOX_BYTES = 32 * 128;             // one 32-row x 128-byte swizzled box
constexpr int C_STAGE_BYTES = 16 * BOX_BYTES;   // the fp32 tile as 4 x 4 boxes of 32 x 32
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + C_STAGE_BYTES + 256;
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
  int tma_epi;              // C (and the split) through the tensor maps cmap, hmap, lmap
  int tri;                  // TRI_* : K blocks a tile can skip (exact zeros of a triangle)
  DevStatus* st;
};
// A triangular operand makes part of each tile's K range exact zeros: with
// TRI_K_FROM_COL, B'[c][k] = 0 for k < c (B' upper), so a tile needs k >= col0; with
// TRI_K_TO_ROW, A'[r][k] = 0 for k > r (A' lower), so it needs k < row0 + BM.  The skipped
// 64-blocks contribute nothing, so every tile keeps at least one block.
constexpr int TRI_K_FROM_COL = 1, TRI_K_TO_ROW = 2;

// byte offset of 16-byte chunk q of row r in a 128-byte-swizzled box (1024-aligned base)
__device__ __forceinline__ uint32_t sw128_off(int r, int q) {
  return (uint32_t)(r * 128 + ((q ^ (r & 7)) << 4));
}

__global__ void __launch_bounds__(256, 1)
    k_gemm_tc(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap bmap,
              const __grid_constant__ CUtensorMap cmap, const __grid_constant__ CUtensorMap hmap,
              const __grid_constant__ CUtensorMap lmap, const GemmTcArgs a) {
  using namespace gt;
  pdl_enter();
  const int tn = blockIdx.x, tm = blockIdx.y, z = blockIdx.z;
  const int row0 = tm * BM, col0 = tn * BN;
  if (a.lower_only && col0 > row0 + BM - 1) return;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* cst = smem + STAGES * STAGE_BYTES;  // C staging (tma_epi)
  uint64_t* bars = reinterpret_cast<uint64_t*>(cst + C_STAGE_BYTES);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;
  uint64_t* drain = accf + 1;
  uint64_t* cbar = drain + 1;  // [8] beta C of each epilogue warp
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(cbar + 8);
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
    mbar_init(accf, 1);
    mbar_init(drain, 1);
    for (int w = 0; w < 8; ++w) mbar_init(&cbar[w], 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (*skip_flag) return;
  // epilogue geometry (tma_epi): TMEM lane quarter wq, column half ch
  const int wq = warp & 3, ch = warp >> 2;
  const bool load_c = a.tma_epi && a.beta != 0.f;
  if (load_c && lane == 0) {
    // beta C for this warp's two 32 x 32 blocks, in flight during the MMAs
    mbar_arrive_expect_tx(&cbar[warp], 2 * BOX_BYTES);
    for (int h = 0; h < 2; ++h) {
      const int cb = 2 * ch + h;
      tma_load_3d(cst + (wq * 4 + cb) * BOX_BYTES, &cmap, &cbar[warp], col0 + 32 * cb,
                  row0 + 32 * wq, z);
    }
  }
  if (warp == 2) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  int kb_lo = (a.tri & TRI_K_FROM_COL) ? col0 / BK : 0;
  int kb_hi = a.kseg_blocks;
  if (a.tri & TRI_K_TO_ROW) kb_hi = min(kb_hi, (row0 + BM + BK - 1) / BK);
  if (kb_lo > kb_hi - 1) kb_lo = kb_hi - 1;
  const int nkb = kb_hi - kb_lo;  // 64-blocks of each segment
  const int nk = a.nseg * nkb;
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
      const int seg = it / nkb, kb = kb_lo + it - seg * nkb;
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
  }
  __syncwarp();

  if (a.tma_epi) {
    bool ok = mbar_wait(accf, 0, abort_flag, kGemmWaitNs);
    if (ok && load_c) ok = mbar_wait(&cbar[warp], 0, abort_flag, kGemmWaitNs);
    if (ok) {
      tc_fence_after();
      // every MMA has completed (accf): stages 0-1 hold the split boxes
      // [hi/lo][column half][lane quarter]
      uint8_t* hbox = smem + (ch * 4 + wq) * BOX_BYTES;
      uint8_t* lbox = smem + (8 + ch * 4 + wq) * BOX_BYTES;
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        const int cb = 2 * ch + h;
        uint8_t* cbox = cst + (wq * 4 + cb) * BOX_BYTES;
        float v[32];
        tmem_ld32(tmem + ((uint32_t)(wq * 32) << 16) + cb * 32, v);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          float4* cp = reinterpret_cast<float4*>(cbox + sw128_off(lane, q));
          float4 r;
          if (load_c) {
            const float4 pv = *cp;
            r = make_float4(fmaf(a.beta, pv.x, a.alpha * v[4 * q]),
                            fmaf(a.beta, pv.y, a.alpha * v[4 * q + 1]),
                            fmaf(a.beta, pv.z, a.alpha * v[4 * q + 2]),
                            fmaf(a.beta, pv.w, a.alpha * v[4 * q + 3]));
          } else {
            r = make_float4(a.alpha * v[4 * q], a.alpha * v[4 * q + 1], a.alpha * v[4 * q + 2],
                            a.alpha * v[4 * q + 3]);
          }
          *cp = r;
          v[4 * q] = r.x, v[4 * q + 1] = r.y, v[4 * q + 2] = r.z, v[4 * q + 3] = r.w;
        }
        if (a.split_out) {
          // 32 bf16 = 64 bytes: chunks 4h .. 4h+3 of the row
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint32_t hw[4], lw[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float x0 = v[8 * q + 2 * e], x1 = v[8 * q + 2 * e + 1];
              const __nv_bfloat16 h0 = __float2bfloat16_rn(x0), h1 = __float2bfloat16_rn(x1);
              const __nv_bfloat16 l0 = __float2bfloat16_rn(x0 - __bfloat162float(h0));
              const __nv_bfloat16 l1 = __float2bfloat16_rn(x1 - __bfloat162float(h1));
              hw[e] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
              lw[e] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
            }
            *reinterpret_cast<uint4*>(hbox + sw128_off(lane, 4 * h + q)) =
                make_uint4(hw[0], hw[1], hw[2], hw[3]);
            *reinterpret_cast<uint4*>(lbox + sw128_off(lane, 4 * h + q)) =
                make_uint4(lw[0], lw[1], lw[2], lw[3]);
          }
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        for (int h = 0; h < 2; ++h) {
          const int cb = 2 * ch + h;
          tma_store_3d(&cmap, cst + (wq * 4 + cb) * BOX_BYTES, col0 + 32 * cb, row0 + 32 * wq, z);
        }
        if (a.split_out) {
          tma_store_3d(&hmap, hbox, col0 + 64 * ch, row0 + 32 * wq, z);
          tma_store_3d(&lmap, lbox, col0 + 64 * ch, row0 + 32 * wq, z);
        }
        bulk_commit_group();
        bulk_wait_read_all();
      }
      __syncwarp();
      tc_fence_before();
    } else if (lane == 0) {
      *abort_flag = 1;
      raise_error(a.st, FFH_ERR_TIMEOUT, 23);
      // this warp's beta-C copy may still be in flight: let it land (bounded) before the
      // CTA's shared memory is released
      if (load_c) {
        volatile int never = 0;
        mbar_wait(&cbar[warp], 0, &never, kGemmWaitNs);
      }
    }
  } else if (warp >= 4) {
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

// 3-D tensor map {cols, rows, batch} with 128-byte swizzled boxes of 32 rows x 128 bytes
// (32 fp32 or 64 bf16 columns); strides in elements.  False where TMA cannot address the
// layout (bases and strides must be 16-byte multiples).
static bool map_epi_3d(CUtensorMap* m, const void* base, bool bf16, uint64_t cols,
                       uint64_t rows, uint64_t batch, uint64_t ld, uint64_t zstride) {
  const uint64_t es = bf16 ? 2 : 4;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (ld * es) % 16) return false;
  if (batch > 1 && (zstride * es) % 16) return false;
  auto fn = encode_fn_chol();
  if (!fn) return false;
  if (batch == 1) zstride = (rows * ld + 7) / 8 * 8;  // unused; any valid stride
  cuuint64_t dims[3] = {cols, rows, batch};
  cuuint64_t strides[2] = {ld * es, zstride * es};
  cuuint32_t box[3] = {(cuuint32_t)(128 / es), 32, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3,
            const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

static cudaError_t gemm_tc(const Split& A, const Split& B, int nseg, const int a_seg[3],
                           const int b_seg[3], int kseg, float* C, int64_t ldc, int64_t strideC,
                           int M, int N, float alpha, float beta, bool lower_only, int batch,
                           DevStatus* st, cudaStream_t s, const Split* out_split = nullptr,
                           int tri = 0) {
  if (M <= 0 || N <= 0 || batch <= 0) return cudaSuccess;
  CUtensorMap am, bm, cm{}, hm{}, lm{};
  if (!map_bf16_kmajor(&am, A.p, (uint64_t)2 * A.kpad, (uint64_t)A.rows_pad * A.batch,
                       (uint64_t)2 * A.kpad, gt::BM))
    return cudaErrorInvalidValue;
  if (!map_bf16_kmajor(&bm, B.p, (uint64_t)2 * B.kpad, (uint64_t)B.rows_pad * B.batch,
                       (uint64_t)2 * B.kpad, gt::BN))
    return cudaErrorInvalidValue;
  bool tma_epi = map_epi_3d(&cm, C, false, (uint64_t)N, (uint64_t)M, (uint64_t)batch,
                            (uint64_t)ldc, (uint64_t)strideC);
  if (tma_epi && out_split) {
    const uint64_t pitch = (uint64_t)2 * out_split->kpad;
    const uint64_t zs = (uint64_t)out_split->rows_pad * pitch;
    tma_epi = map_epi_3d(&hm, out_split->p, true, (uint64_t)N, (uint64_t)M, (uint64_t)batch,
                         pitch, zs) &&
              map_epi_3d(&lm, out_split->p + out_split->kpad, true, (uint64_t)N, (uint64_t)M,
                         (uint64_t)batch, pitch, zs);
  }
  static PerDeviceOnce attr;
  {
    cudaError_t e = smem_attr_once((const void*)k_gemm_tc, gt::SMEM_BYTES, attr);
    if (e != cudaSuccess) return e;
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
  g.tma_epi = tma_epi ? 1 : 0;
  g.tri = tri;
  g.st = st;
  dim3 grid((N + gt::BN - 1) / gt::BN, (M + gt::BM - 1) / gt::BM, batch);
  cudaError_t e = launch_pdl(k_gemm_tc, grid, dim3(256), gt::SMEM_BYTES, s, am, bm, cm, hm, lm, g);
  note_launches(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Persistent trailing update C -= A' A'^T over the lower 128 x 128 tiles of an M x M block
// (the columns beyond the next column block, on the side stream).  Each CTA walks its tiles
// (t = blockIdx.x, + gridDim.x, ...) through one pipeline: the producer streams A' rows of
// the tile's row and column blocks, the MMA issuer alternates two 128-column TMEM
// accumulators, and the four epilogue warps drain tile j (C = alpha acc + beta C through
// swizzled shared memory and TMA stores, each warp its 32 rows) while tile j+1's MMAs run.
// Each epilogue warp loads its rows of the next tile's C as soon as its stores have read
// the staging buffer.  C must be TMA-addressable (16-byte aligned rows).
// ---------------------------------------------------------------------------
namespace sy {
constexpr int BM = 128, BN = 128, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2, B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int BOX = 32 * 128;           // 32 rows x 128 bytes (32 fp32)
constexpr int WARP_C = 4 * BOX;         // an epilogue warp's 32 rows x 128 columns
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + 4 * WARP_C + 256;
constexpr uint32_t TMEM_COLS = 256;     // two 128-column accumulators
}  // namespace sy

struct SyrkArgs {
  int ntiles;               // lower tiles: ntm (ntm + 1) / 2 for ntm = ceil(M / 128)
  int nseg, kseg_blocks;    // K segments, 64-blocks per segment
  int a_off[3], b_off[3];   // x offsets of the segments for the row / column operand
  float alpha, beta;
  DevStatus* st;
};

__global__ void __launch_bounds__(256, 1)
    k_syrk_tc(const __grid_constant__ CUtensorMap amap, const __grid_constant__ CUtensorMap cmap,
              const SyrkArgs a) {
  using namespace sy;
  pdl_enter();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* cst = smem + STAGES * STAGE_BYTES;  // [epilogue warp][4 boxes]
  uint64_t* bars = reinterpret_cast<uint64_t*>(cst + 4 * WARP_C);
  uint64_t* full = bars;
  uint64_t* empty = bars + STAGES;
  uint64_t* accf = bars + 2 * STAGES;  // [2]
  uint64_t* acce = accf + 2;           // [2]
  uint64_t* cbar = acce + 2;           // [4]
  uint64_t* drain = cbar + 4;
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
      mbar_init(&acce[b], 4);
    }
    for (int w = 0; w < 4; ++w) mbar_init(&cbar[w], 1);
    mbar_init(drain, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (*skip_flag) return;
  const int wq = warp - 4;
  if (warp >= 4 && lane == 0 && (int)blockIdx.x < a.ntiles) {
    // the first tile's C rows of this epilogue warp
    int tm, tn;
    lower_tile(blockIdx.x, tm, tn);
    mbar_arrive_expect_tx(&cbar[wq], WARP_C);
    for (int cb = 0; cb < 4; ++cb)
      tma_load_3d(cst + wq * WARP_C + cb * BOX, &cmap, &cbar[wq], tn * BN + 32 * cb,
                  tm * BM + 32 * wq, 0);
  }
  if (warp == 2) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int nk = a.nseg * a.kseg_blocks;

  if (warp == 0 && lane == 0) {
    bool ok = true;
    int it = 0;
    for (int t = blockIdx.x; t < a.ntiles && ok; t += gridDim.x) {
      int tm, tn;
      lower_tile(t, tm, tn);
      for (int i = 0; i < nk; ++i, ++it) {
        const int s = it % STAGES;
        const uint32_t ph = (it / STAGES) & 1;
        if (!mbar_wait(&empty[s], ph ^ 1, abort_flag, kGemmWaitNs)) {
          ok = false;
          break;
        }
        const int seg = i / a.kseg_blocks, kb = i - seg * a.kseg_blocks;
        mbar_arrive_expect_tx(&full[s], STAGE_BYTES);
        uint8_t* sa = smem + s * STAGE_BYTES;
        tma_load_2d(sa, &amap, &full[s], a.a_off[seg] + kb * BK, tm * BM);
        tma_load_2d(sa + A_BYTES, &amap, &full[s], a.b_off[seg] + kb * BK, tn * BN);
      }
    }
    if (!ok) {
      *abort_flag = 1;
      raise_error(a.st, FFH_ERR_TIMEOUT, 25);
    }
    const int first = it > STAGES ? it - STAGES : 0;
    for (int j = first; j < it; ++j) {
      volatile int never = 0;
      mbar_wait(&full[j % STAGES], (j / STAGES) & 1, &never, kGemmWaitNs);
    }
  } else if (warp == 1 && lane == 0) {
    constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, false, false);
    bool ok = true;
    int it = 0, j = 0;
    for (int t = blockIdx.x; t < a.ntiles && ok; t += gridDim.x, ++j) {
      const int buf = j & 1;
      if (!mbar_wait(&acce[buf], ((j >> 1) & 1) ^ 1, abort_flag, kGemmWaitNs)) {
        ok = false;
        break;
      }
      tc_fence_after();
      for (int i = 0; i < nk; ++i, ++it) {
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
          mma_bf16(tmem + buf * BN, sw128_desc(sa + k * 32, 16, 1024),
                   sw128_desc(sb + k * 32, 16, 1024), idesc, (i > 0 || k > 0) ? 1u : 0u);
        mma_commit(&empty[s]);
      }
      if (!ok) break;
      mma_commit(&accf[buf]);
    }
    if (!ok) {
      *abort_flag = 1;
      raise_error(a.st, FFH_ERR_TIMEOUT, 26);
    }
    mma_commit(drain);
    volatile int never = 0;
    mbar_wait(drain, 0, &never, kGemmWaitNs);
  } else if (warp >= 4) {
    uint8_t* wc = cst + wq * WARP_C;
    int j = 0;
    for (int t = blockIdx.x; t < a.ntiles; t += gridDim.x, ++j) {
      const int buf = j & 1;
      int tm, tn;
      lower_tile(t, tm, tn);
      bool ok = mbar_wait(&cbar[wq], j & 1, abort_flag, kGemmWaitNs);
      if (ok) ok = mbar_wait(&accf[buf], (j >> 1) & 1, abort_flag, kGemmWaitNs);
      if (!ok) {
        if (lane == 0) {
          *abort_flag = 1;
          raise_error(a.st, FFH_ERR_TIMEOUT, 27);
          // this tile's C copy may still be in flight: let it land (bounded) before the
          // CTA's shared memory is released
          volatile int never = 0;
          mbar_wait(&cbar[wq], j & 1, &never, kGemmWaitNs);
        }
        break;
      }
      tc_fence_after();
#pragma unroll 1
      for (int cb = 0; cb < 4; ++cb) {
        float v[32];
        tmem_ld32(tmem + ((uint32_t)(wq * 32) << 16) + buf * BN + cb * 32, v);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          float4* cp = reinterpret_cast<float4*>(wc + cb * BOX + sw128_off(lane, q));
          const float4 pv = *cp;
          *cp = make_float4(fmaf(a.beta, pv.x, a.alpha * v[4 * q]),
                            fmaf(a.beta, pv.y, a.alpha * v[4 * q + 1]),
                            fmaf(a.beta, pv.z, a.alpha * v[4 * q + 2]),
                            fmaf(a.beta, pv.w, a.alpha * v[4 * q + 3]));
        }
      }
      // this warp's reads of the accumulator are done
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acce[buf]);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        for (int cb = 0; cb < 4; ++cb)
          tma_store_3d(&cmap, wc + cb * BOX, tn * BN + 32 * cb, tm * BM + 32 * wq, 0);
        bulk_commit_group();
        bulk_wait_read_all();
        const int tnext = t + gridDim.x;
        if (tnext < a.ntiles) {
          int tm2, tn2;
          lower_tile(tnext, tm2, tn2);
          mbar_arrive_expect_tx(&cbar[wq], WARP_C);
          for (int cb = 0; cb < 4; ++cb)
            tma_load_3d(wc + cb * BOX, &cmap, &cbar[wq], tn2 * BN + 32 * cb, tm2 * BM + 32 * wq,
                        0);
        }
      }
      __syncwarp();
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

// C (M x M, pitch ldc) -= A' A'^T on the lower tiles, A' = the split rows of A.  Returns
// cudaErrorNotSupported when C's layout is not TMA-addressable (the caller then uses
// gemm_tc).  grid_cap bounds the persistent CTAs (SMs left to the other stream).
static cudaError_t syrk_tc(const Split& A, const int a_seg[3], const int b_seg[3], int nseg,
                           int kseg, float* C, int64_t ldc, int M, float alpha, float beta,
                           int grid_cap, DevStatus* st, cudaStream_t s) {
  if (M <= 0) return cudaSuccess;
  CUtensorMap am, cm;
  if (!map_epi_3d(&cm, C, false, (uint64_t)M, (uint64_t)M, 1, (uint64_t)ldc, 0))
    return cudaErrorNotSupported;
  if (!map_bf16_kmajor(&am, A.p, (uint64_t)2 * A.kpad, (uint64_t)A.rows_pad * A.batch,
                       (uint64_t)2 * A.kpad, sy::BM))
    return cudaErrorInvalidValue;
  static PerDeviceOnce attr;
  {
    cudaError_t e = smem_attr_once((const void*)k_syrk_tc, sy::SMEM_BYTES, attr);
    if (e != cudaSuccess) return e;
  }
  SyrkArgs g{};
  const int ntm = (M + sy::BM - 1) / sy::BM;
  g.ntiles = ntm * (ntm + 1) / 2;
  g.nseg = nseg;
  g.kseg_blocks = (kseg + sy::BK - 1) / sy::BK;
  for (int i = 0; i < 3; ++i) {
    g.a_off[i] = a_seg[i];
    g.b_off[i] = b_seg[i];
  }
  g.alpha = alpha;
  g.beta = beta;
  g.st = st;
  const int grid = std::max(1, std::min(g.ntiles, grid_cap));
  cudaError_t e = launch_pdl(k_syrk_tc, dim3(grid), dim3(256), sy::SMEM_BYTES, s, am, cm, g);
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
// One 64 x 64 tile of (r, c) per block, staged through shared memory so that the source
// is read along its contiguous dimension in both orientations; each thread then writes
// four consecutive columns of hi and of lo (8 bytes each).
constexpr int SPLIT_TILE = 64;
__global__ void __launch_bounds__(256) k_split_hilo(const float* __restrict__ src, int64_t lds,
                                                    int64_t src_stride, int rows, int cols,
                                                    int trans, __nv_bfloat16* __restrict__ dst,
                                                    int rows_pad, int kpad,
                                                    const DevStatus* gate) {
  pdl_enter();
  if (gated_off(gate)) return;
  __shared__ float tile[SPLIT_TILE][SPLIT_TILE + 1];
  const int z = blockIdx.z;
  const int r0 = blockIdx.y * SPLIT_TILE, c0 = blockIdx.x * SPLIT_TILE;
  const float* sz = src + (int64_t)z * src_stride;
  const int t = threadIdx.x;
  const int f = t & 63, g = t >> 6;  // fast (contiguous) and slow index of the source read
#pragma unroll 4
  for (int i = 0; i < SPLIT_TILE / 4; ++i) {
    const int sl = g + 4 * i;
    if (!trans) {
      const int r = r0 + sl, c = c0 + f;
      tile[sl][f] = (r < rows && c < cols) ? sz[(int64_t)r * lds + c] : 0.f;
    } else {
      const int r = r0 + f, c = c0 + sl;  // view (r, c) = source row c, column r
      tile[f][sl] = (r < rows && c < cols) ? sz[(int64_t)c * lds + r] : 0.f;
    }
  }
  __syncthreads();
  const int cq = (t & 15) * 4;
#pragma unroll 4
  for (int i = 0; i < SPLIT_TILE / 16; ++i) {
    const int rr = (t >> 4) + 16 * i;
    __nv_bfloat16 hi[4], lo[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float x = tile[rr][cq + e];
      hi[e] = __float2bfloat16_rn(x);
      lo[e] = __float2bfloat16_rn(x - __bfloat162float(hi[e]));
    }
    __nv_bfloat16* drow = dst + ((int64_t)z * rows_pad + r0 + rr) * (2 * (int64_t)kpad);
    *reinterpret_cast<uint2*>(drow + c0 + cq) = *reinterpret_cast<const uint2*>(hi);
    *reinterpret_cast<uint2*>(drow + kpad + c0 + cq) = *reinterpret_cast<const uint2*>(lo);
  }
}

static cudaError_t split(const float* src, int64_t lds, int64_t src_stride, int rows, int cols,
                         bool trans, const Split& d, cudaStream_t s) {
  if ((int64_t)d.rows_pad * d.kpad * d.batch == 0) return cudaSuccess;
  // rows_pad (a multiple of 128) and kpad (a multiple of 64) are whole tiles
  const dim3 grid((unsigned)(d.kpad / SPLIT_TILE), (unsigned)(d.rows_pad / SPLIT_TILE),
                  (unsigned)d.batch);
  cudaError_t e = launch_pdl(k_split_hilo, grid, dim3(256), 0, s, src, lds, src_stride, rows,
                             cols, trans ? 1 : 0, d.p, d.rows_pad, d.kpad, current_gate());
  note_launches(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

// ---------------------------------------------------------------------------
// 128 x 128 diagonal block: Cholesky factor L11 and inverse M11 = L11^-1, one CTA of
// 512 threads (16 warps), blocked by 32 (sub-panels q = 0..3, rows/cols Q = [32q, 32q+32)).
//   A(q)  warp 0 factors the 32 x 32 diagonal block D_q and inverts it in registers:
//         lane i holds row i of D_q and column i of its inverse; the 2 x 2 pivot block
//         of columns j, j+1 is broadcast by shuffle, and the remaining columns shift
//         down two registers per step so every register index is static.  Writes L_qq,
//         Mi_q = L_qq^-1 and Mt[x][k] = Mi_q[k][x].
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
// Outputs: L11 and M11 (fp32; their destinations arrive zeroed, so only the lower
// triangle is stored) and the bf16 hi/lo split of M11 ([hi | lo] rows, pitch 256, dense),
// the B operand of the panel GEMM.
// ---------------------------------------------------------------------------
constexpr int LB = 128;
constexpr int LP = LB + 1;   // pitch of the row-major 128 x 128 blocks (conflict-free columns)
constexpr int PTP = LB + 4;  // pitch of Pt (float4 rows)
constexpr int MP = LB + 4;   // pitch of M11 (float4 rows)
constexpr int MTP = 36;      // pitch of Mt
constexpr int TP = 100;      // pitch of the 32 x 96 scratch T
constexpr int LEAF_THREADS = 512;
// float offsets of the regions of the kernel's dynamic shared memory
constexpr int OFF_LS = 0;                          // [LB][LP]  working block -> L11
constexpr int OFF_MS = OFF_LS + LB * LP;           // [LB][MP]  M11
constexpr int OFF_PT = OFF_MS + LB * MP;           // [2][32][PTP] transposed sub-panels
constexpr int OFF_MT = OFF_PT + 2 * 32 * PTP;      // [2][32][MTP] diagonal-block inverses^T
constexpr int OFF_T = OFF_MT + 2 * 32 * MTP;       // [32][TP]
constexpr int OFF_PIV = OFF_T + 32 * TP;           // [LB] pivots
constexpr int OFF_LBUF = OFF_PIV + LB;             // [2][32][2] pair broadcast (warp 0)
constexpr int LB_SMEM = (OFF_LBUF + 128) * 4 + 64;

// A(q): factor and invert the diagonal block (warp 0 only); the pivots go to pivs[c0..].
// Two columns per step: every lane forms the 2 x 2 pivot block of columns j, j+1
// (three shuffles from lanes j, j+1), its own entries l_{lane,j}, l_{lane,j+1} and the
// matching rows j, j+1 of the inverse, then applies the rank-2 update to its row (and to
// its column of the inverse) with packed two-wide fp32 FMAs (per component the same
// rounding as fmaf).  The two updates of an entry are applied one after the other, in
// the same order and rounding as two one-column steps.  The pairs (l_j, l_{j+1}) reach
// the other lanes through a shared buffer written rotated (slot s = (lane - j - 2) mod 32
// holds lane lane's pair), laid out so that one broadcast float4 gives the l_j of slots
// 2g, 2g+1 followed by their l_{j+1}; the buffer alternates by the parity of j / 2, so one
// warp barrier per step suffices.  Look-ahead by one step: as soon as step j has updated
// columns j+2, j+3, the pivot block of step j+2 is factored in registers while the rest
// of step j's update runs, and published (stores) after it, so the pivot chain (shuffles,
// two reciprocal square roots) overlaps the update.  Pivot tests are branch-free selects
// (a failed pivot is replaced by 1 and reported once after the sweep).  Not inlined: one
// copy serves the four sub-panels.
struct PivotPair {
  float l0, l1, m0, m1, p00, q11;
  bool bad0, bad1;
};

// The 2 x 2 pivot block of columns j, j+1 and this lane's entries (registers only).
__device__ __forceinline__ PivotPair leaf_pivot_pair(float p00, float p10, float p11, float2 a0,
                                                     float2 mc0) {
  PivotPair p;
  // the tests are warp-uniform (broadcast values)
  p.bad0 = !(p00 > 0.f) | !isfinite(p00);
  p00 = p.bad0 ? 1.f : p00;
  // 1/sqrt to within 2 ulp; far below the fp32 accumulation error of the updates
  const float r0 = rsqrtf(p00);
  const float l10 = p10 * r0;  // l_{j+1,j}
  float q11 = fmaf(-l10, l10, p11);
  p.bad1 = !(q11 > 0.f) | !isfinite(q11);
  q11 = p.bad1 ? 1.f : q11;
  const float r1 = rsqrtf(q11);
  p.p00 = p00;
  p.q11 = q11;
  p.l0 = a0.x * r0;                     // lane > j: l_{lane,j}; lane j: sqrt(p00)
  p.l1 = fmaf(-p.l0, l10, a0.y) * r1;   // lane > j+1: l_{lane,j+1}; lane j+1: diagonal
  p.m0 = mc0.x * r0;                    // Mi[j][lane]
  p.m1 = fmaf(-l10, p.m0, mc0.y) * r1;  // Mi[j+1][lane]
  return p;
}

// Publish step j's pair: the rotated broadcast buffer, L, M11, Mt and the pivots.
__device__ __forceinline__ void leaf_pivot_store(const PivotPair& p, int j, int c0, float* Ls,
                                                 float* Ms, float* Mt, float* lbuf, float* pivs,
                                                 int& first_bad) {
  const int lane = threadIdx.x & 31;
  first_bad = (first_bad < 0 && p.bad0) ? j : first_bad;
  first_bad = (first_bad < 0 && p.bad1) ? j + 1 : first_bad;
  float* lb = lbuf + ((j >> 1) & 1) * 64;
  const int slot = (lane - j - 2) & 31;
  lb[4 * (slot >> 1) + (slot & 1)] = p.l0;
  lb[4 * (slot >> 1) + 2 + (slot & 1)] = p.l1;
  if (lane == 0) {
    pivs[c0 + j] = p.p00;
    pivs[c0 + j + 1] = p.q11;
  }
  Ls[(c0 + lane) * LP + c0 + j] = lane >= j ? p.l0 : 0.f;
  Ls[(c0 + lane) * LP + c0 + j + 1] = lane >= j + 1 ? p.l1 : 0.f;
  Ms[(c0 + j) * MP + c0 + lane] = p.m0;
  Ms[(c0 + j + 1) * MP + c0 + lane] = p.m1;
  *reinterpret_cast<float2*>(Mt + lane * MTP + j) = make_float2(p.m0, p.m1);
}

// Register pair k of a lane: columns j+2k, j+2k+1 (of its row of D) and rows j+2k, j+2k+1
// (of its column of the inverse).  Step j's update of pair k (k = 1..15) lands in pair
// k - 1; v holds (l_j, l_j, l_{j+1}, l_{j+1}) of the two rows j+2k, j+2k+1.
__device__ __forceinline__ void leaf_pair_update(float2* a2, float2* mc2, int k, float4 v,
                                                 float2 nl0, float2 nl1, float2 nm0,
                                                 float2 nm1) {
  const float2 v0 = make_float2(v.x, v.y), v1 = make_float2(v.z, v.w);
  a2[k - 1] = __ffma2_rn(nl1, v1, __ffma2_rn(nl0, v0, a2[k]));
  mc2[k - 1] = __ffma2_rn(v1, nm1, __ffma2_rn(v0, nm0, mc2[k]));
}

__device__ __noinline__ void leaf_diag(int mt_off, int c0, int64_t o, DevStatus* st,
                                          bool& bad) {
  // the regions are addressed from the kernel's shared array (not through pointer
  // arguments), so every access compiles to a shared-memory instruction
  extern __shared__ float sh[];
  float* Ls = sh + OFF_LS;
  float* Ms = sh + OFF_MS;
  float* Mt = sh + mt_off;
  float* lbuf = sh + OFF_LBUF;
  float* pivs = sh + OFF_PIV;
  const int lane = threadIdx.x & 31;
  constexpr unsigned FULL = 0xffffffffu;
  float2 a2[16], mc2[16];
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    a2[k].x = (2 * k <= lane) ? Ls[(c0 + lane) * LP + c0 + 2 * k] : 0.f;
    a2[k].y = (2 * k + 1 <= lane) ? Ls[(c0 + lane) * LP + c0 + 2 * k + 1] : 0.f;
    mc2[k].x = (2 * k == lane) ? 1.f : 0.f;
    mc2[k].y = (2 * k + 1 == lane) ? 1.f : 0.f;
  }
  int first_bad = -1;
  PivotPair p = leaf_pivot_pair(__shfl_sync(FULL, a2[0].x, 0), __shfl_sync(FULL, a2[0].x, 1),
                                __shfl_sync(FULL, a2[0].y, 1), a2[0], mc2[0]);
  leaf_pivot_store(p, 0, c0, Ls, Ms, Mt, lbuf, pivs, first_bad);
  __syncwarp();
#pragma unroll 1
  for (int j = 0; j < 30; j += 2) {
    const float4* lb4 = reinterpret_cast<const float4*>(lbuf + ((j >> 1) & 1) * 64);
    const float2 nl0 = make_float2(-p.l0, -p.l0), nl1 = make_float2(-p.l1, -p.l1);
    const float2 nm0 = make_float2(-p.m0, -p.m0), nm1 = make_float2(-p.m1, -p.m1);
    // pairs past the block (rows j + 2k > 31) only reach registers shifted past the block
    leaf_pair_update(a2, mc2, 1, lb4[0], nl0, nl1, nm0, nm1);
    // step j+2's pivot block, in registers only: no shared-memory store comes between the
    // broadcast loads below and the chain, so the two overlap
    const PivotPair pn =
        leaf_pivot_pair(__shfl_sync(FULL, a2[0].x, j + 2), __shfl_sync(FULL, a2[0].x, j + 3),
                        __shfl_sync(FULL, a2[0].y, j + 3), a2[0], mc2[0]);
#pragma unroll
    for (int k = 2; k < 16; ++k) leaf_pair_update(a2, mc2, k, lb4[k - 1], nl0, nl1, nm0, nm1);
    a2[15] = make_float2(0.f, 0.f);
    mc2[15] = make_float2(0.f, 0.f);
    // every lane has read step j's buffer; step j+2 writes the other one
    leaf_pivot_store(pn, j + 2, c0, Ls, Ms, Mt, lbuf, pivs, first_bad);
    p = pn;
    __syncwarp();
  }
  if (first_bad >= 0) {
    if (lane == 0 && !bad) raise_error(st, FFH_ERR_NOT_SPD, (int)(o + c0 + first_bad));
    bad = true;
  }
}

// acc[0..1] += a * (b.x, b.y), (b.z, b.w): one row of a 4-wide register block in two
// packed fp32 FMAs (per component the same rounding as fmaf)
__device__ __forceinline__ void fma_row4(float2* acc, float a, float4 b) {
  const float2 aa = make_float2(a, a);
  acc[0] = __ffma2_rn(aa, make_float2(b.x, b.y), acc[0]);
  acc[1] = __ffma2_rn(aa, make_float2(b.z, b.w), acc[1]);
}

// Rank-32 update of one 4 x 4 block of the trailing lower triangle from the transposed
// sub-panel: A[r][c] -= sum_k Pt[k][r] Pt[k][c].
__device__ __forceinline__ void leaf_trail_block(float* Ls, const float* Pt, int r0, int cc0) {
  float2 acc[4][2] = {};
#pragma unroll 8
  for (int k = 0; k < 32; ++k) {
    const float4 av = *reinterpret_cast<const float4*>(Pt + k * PTP + r0);
    const float4 bv = *reinterpret_cast<const float4*>(Pt + k * PTP + cc0);
    fma_row4(acc[0], av.x, bv);
    fma_row4(acc[1], av.y, bv);
    fma_row4(acc[2], av.z, bv);
    fma_row4(acc[3], av.w, bv);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float ac[4] = {acc[i][0].x, acc[i][0].y, acc[i][1].x, acc[i][1].y};
#pragma unroll
    for (int jx = 0; jx < 4; ++jx)
      if (cc0 + jx <= r0 + i) Ls[(r0 + i) * LP + cc0 + jx] -= ac[jx];
  }
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
    float2 acc[2][2] = {};
    // M lower triangular: M[k][x] = 0 for k < x, so k starts at x0
    for (int k = x0; k < c0; ++k) {
      const float4 bv = *reinterpret_cast<const float4*>(Ms + k * MP + x0);
#pragma unroll
      for (int i = 0; i < 2; ++i) fma_row4(acc[i], Ls[(c0 + i0 + i) * LP + k], bv);
    }
#pragma unroll
    for (int i = 0; i < 2; ++i)
      *reinterpret_cast<float4*>(T + (i0 + i) * TP + x0) =
          make_float4(acc[i][0].x, acc[i][0].y, acc[i][1].x, acc[i][1].y);
  }
}

__device__ __forceinline__ void leaf_inverse_apply(float* Ms, const float* T, int c0, int t,
                                                   int nt) {
  const int nbx = c0 / 4;
  // 2 rows x 4 columns per thread
  for (int blk = t; blk < 16 * nbx; blk += nt) {
    const int i0 = (blk / nbx) * 2, x0 = (blk % nbx) * 4;
    float2 acc[2][2] = {};
    // Mi lower triangular: row i needs j <= i < i0 + 2
    for (int j = 0; j < i0 + 2; ++j) {
      const float4 bv = *reinterpret_cast<const float4*>(T + j * TP + x0);
#pragma unroll
      for (int i = 0; i < 2; ++i) fma_row4(acc[i], Ms[(c0 + i0 + i) * MP + c0 + j], bv);
    }
#pragma unroll
    for (int i = 0; i < 2; ++i)
      *reinterpret_cast<float4*>(Ms + (c0 + i0 + i) * MP + x0) =
          make_float4(-acc[i][0].x, -acc[i][0].y, -acc[i][1].x, -acc[i][1].y);
  }
}

__global__ void __launch_bounds__(LEAF_THREADS, 1) k_chol_leaf(float* W, int64_t ldw, int64_t d,
                                                               int64_t o, float* L, int64_t ldl,
                                                               float* Minv, int64_t ldm,
                                                               __nv_bfloat16* m11_split,
                                                               DevStatus* st, int fault) {
  extern __shared__ float sh[];
  float* Ls = sh + OFF_LS;
  float* Ms = sh + OFF_MS;
  float* Ptb = sh + OFF_PT;
  float* Mtb = sh + OFF_MT;
  float* T = sh + OFF_T;
  float* pivs = sh + OFF_PIV;
  pdl_enter();
  // the fit this factorization belongs to has failed or stopped at its tolerance
  if (gated_off(st)) return;
  const int b = (int)((d - o) < LB ? (d - o) : LB);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // the lower triangle of the block, all loads of a thread in flight together
  constexpr int NLD = LB * LB / 4 / LEAF_THREADS;
  float4 v[NLD];
#pragma unroll
  for (int u = 0; u < NLD; ++u) {
    const int idx = tid + u * LEAF_THREADS;
    const int i = idx >> 5, j4 = (idx & 31) * 4;
    v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i < b && j4 <= i) {
      const float* src = W + (o + i) * ldw + o + j4;
      if (j4 + 3 < b && (((uintptr_t)src) & 15) == 0) {
        v[u] = *reinterpret_cast<const float4*>(src);
      } else {
        if (j4 + 0 < b) v[u].x = src[0];
        if (j4 + 1 < b) v[u].y = src[1];
        if (j4 + 2 < b) v[u].z = src[2];
        if (j4 + 3 < b) v[u].w = src[3];
      }
    }
  }
#pragma unroll
  for (int u = 0; u < NLD; ++u) {
    const int idx = tid + u * LEAF_THREADS;
    const int i = idx >> 5, j4 = (idx & 31) * 4;
    const float vv[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
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
  if (warp == 0) leaf_diag(OFF_MT, 0, o, st, bad);
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
    float2 acc2[4][2] = {};
    if (has) {
      for (int x = 0; x < k0 + 4; ++x) {  // Mi[k][x] = 0 for x > k
        const float4 bv = *reinterpret_cast<const float4*>(Mt + x * MTP + k0);
#pragma unroll
        for (int i = 0; i < 4; ++i) fma_row4(acc2[i], Ls[(r0 + i) * LP + c0 + x], bv);
      }
    }
    __syncthreads();
    if (has) {
      float acc[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        acc[i][0] = acc2[i][0].x, acc[i][1] = acc2[i][0].y;
        acc[i][2] = acc2[i][1].x, acc[i][3] = acc2[i][1].y;
      }
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
          leaf_diag(OFF_MT + ((q + 1) & 1) * 32 * MTP, c0 + 32, o, st, bad);
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
    // L and Minv arrive zeroed: groups entirely above the diagonal are not stored
    if (i < b && j0 <= i) {
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

// M = L^-1 by recursive doubling over block size b = 128, 256, ... (the 128 x 128 diagonal
// blocks of M already hold the leaf kernels' inverses); T and the split buffers are scratch.
// From this order on the look-ahead schedule pairs the panels of the trailing update
// (the fp32 trailing matrix no longer fits in L2, so its traffic bounds the factorization)
constexpr int64_t kGroupedMinD = 8192;

static cudaError_t cholesky_inverse(const float* L, float* Linv, int64_t d, float* T,
                                    __nv_bfloat16* const* sb, DevStatus* st, cudaStream_t s) {
  cudaError_t e;
  if (!Linv) return cudaSuccess;
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
      // B' = M11^T is upper triangular: output column block c needs k >= c
      if ((e = gemm_tc(l21, m11t, 3, as1, bs1, (int)b, T, b, (int64_t)rp * b, rows, (int)b, 1.f,
                       0.f, false, batch, st, s, nullptr, TRI_K_FROM_COL)) != cudaSuccess)
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
      // A' = M22 is lower triangular: output row block r needs k < r + 128
      if ((e = gemm_tc(m22, tt, 3, as2, bs2, rows, Linv + (o + b) * d + o, d, zs, rows, (int)b,
                       -1.f, 0.f, false, batch, st, s, nullptr, TRI_K_TO_ROW)) != cudaSuccess)
        return e;
    }
  }
  return cudaSuccess;
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
  static PerDeviceOnce attr;
  if ((e = smem_attr_once((const void*)k_chol_leaf, LB_SMEM, attr)) != cudaSuccess) return e;
  if ((e = cudaMemcpy2DAsync(W, d * 4, F, ldf * 4, d * 4, d, cudaMemcpyDeviceToDevice, s)) !=
      cudaSuccess)
    return e;
  if ((e = cudaMemsetAsync(L, 0, (size_t)d * d * 4, s)) != cudaSuccess) return e;
  if (Linv && (e = cudaMemsetAsync(Linv, 0, (size_t)d * d * 4, s)) != cudaSuccess) return e;
  if ((e = cudaMemsetAsync(&st->logdet, 0, sizeof(double), s)) != cudaSuccess) return e;
  float* Mdiag = Linv ? Linv : T;  // the diagonal-block inverses (T is free until the inverse)
  const int np = (int)((d + LB - 1) / LB);
  const int aseg[3] = {0, 0, 128}, bseg[3] = {0, 128, 0};
  if (cs && d >= kGroupedMinD) {
    // Panels in pairs: the trailing update beyond the next two column blocks applies both
    // panels at once (K = 256), which halves the passes over the fp32 trailing matrix
    // (the bound at large d) and the waits on the side stream.  The pair's L21 splits share
    // one buffer laid out [hi(256) | lo(256)] per row, rows from the first panel's
    // trailing rows: the first panel's split at K offset 0, the second's at K offset 128
    // and 128 rows down.
    const int gseg[3] = {0, 0, 256}, hseg[3] = {0, 256, 0};
    const int rows_pad_all = (int)((d + 127) / 128 * 128);
    const int64_t pitch = 512;
    for (int p = 0; p < np; ++p) {
      const int64_t o = (int64_t)p * LB;
      if ((e = launch_pdl(k_chol_leaf, dim3(1), dim3(LEAF_THREADS), LB_SMEM, s, W, d, d, o, L, d,
                          Mdiag, d, sb[1], st, fault)) != cudaSuccess)
        return e;
      note_launches(1);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
      const int rows = (int)(d - o - LB);
      if (rows <= 0) continue;
      const bool second = (p & 1) != 0;
      __nv_bfloat16* pair = sb[2 + 2 * ((p >> 1) & 1)];
      // solve: L21 = A21 M11^T, its split into the pair buffer
      Split a21{sb[0] + (size_t)LB * 2 * 128, (int)((rows + 127) / 128 * 128), 128, 1};
      Split m11{sb[1], 128, 128, 1};
      if (p == 0 && (e = split(W + (o + LB) * d + o, d, 0, rows, LB, false, a21, s)) != cudaSuccess)
        return e;
      Split l21{second ? pair + LB * pitch + 128 : pair, rows_pad_all, 256, 1};
      if ((e = gemm_tc(a21, m11, 3, aseg, bseg, 128, L + (o + LB) * d + o, d, 0, rows, LB, 1.f,
                       0.f, false, 1, st, s, &l21)) != cudaSuccess)
        return e;
      const int rows_pad = (rows + 127) / 128 * 128;
      Split next_a21{sb[0], rows_pad + LB, 128, 1};
      if (!second) {
        // the next column block with this panel alone (K = 128), after the previous pair's
        // side update of the columns beyond it
        if (p > 0 && (e = cudaStreamWaitEvent(s, cs->ev[2 + (((p >> 1) - 1) & 1)], 0)) !=
                         cudaSuccess)
          return e;
        Split v{pair, rows_pad_all, 256, 1};
        Split head{pair, LB, 256, 1};
        if ((e = gemm_tc(v, head, 3, gseg, hseg, 128, W + (o + LB) * d + (o + LB), d, 0, rows,
                         rows < LB ? rows : LB, -1.f, 1.f, true, 1, st, s,
                         rows > LB ? &next_a21 : nullptr)) != cudaSuccess)
          return e;
        continue;
      }
      // second panel of the pair: both panels' L21 from this panel's trailing rows on
      Split v{pair + LB * pitch, rows_pad_all - LB, 256, 1};
      Split head{pair + LB * pitch, LB, 256, 1};
      if (rows > LB) {
        // side: the columns beyond the next block, A22[128:, 128:] -= V[128:] V[128:]^T, K = 256
        if ((e = cudaEventRecord(cs->ev[1], s)) != cudaSuccess) return e;
        if ((e = cudaStreamWaitEvent(cs->side, cs->ev[1], 0)) != cudaSuccess) return e;
        Split rest{v.p + LB * pitch, rows_pad_all - 2 * LB, 256, 1};
        float* C22 = W + (o + 2 * LB) * d + (o + 2 * LB);
        const int cap = num_sms() - 24;
        e = syrk_tc(rest, gseg, hseg, 3, 256, C22, d, rows - LB, -1.f, 1.f, cap, st, cs->side);
        if (e == cudaErrorNotSupported)
          e = gemm_tc(rest, rest, 3, gseg, hseg, 256, C22, d, 0, rows - LB, rows - LB, -1.f, 1.f,
                      true, 1, st, cs->side);
        if (e != cudaSuccess) return e;
        if ((e = cudaEventRecord(cs->ev[2 + ((p >> 1) & 1)], cs->side)) != cudaSuccess) return e;
      } else if ((e = cudaEventRecord(cs->ev[2 + ((p >> 1) & 1)], cs->side)) != cudaSuccess) {
        return e;
      }
      // critical: the next column block with both panels (K = 256)
      if ((e = gemm_tc(v, head, 3, gseg, hseg, 256, W + (o + LB) * d + (o + LB), d, 0, rows,
                       rows < LB ? rows : LB, -1.f, 1.f, true, 1, st, s,
                       rows > LB ? &next_a21 : nullptr)) != cudaSuccess)
        return e;
    }
    // the side stream's last update precedes the inverse
    if ((e = cudaEventRecord(cs->ev[2], cs->side)) != cudaSuccess) return e;
    if ((e = cudaStreamWaitEvent(s, cs->ev[2], 0)) != cudaSuccess) return e;
    return cholesky_inverse(L, Linv, d, T, sb, st, s);
  }
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
      float* C22 = W + (o + 2 * LB) * d + (o + 2 * LB);
      // persistent, leaving 24 SMs to the critical stream's kernels (at large d this update
      // is the bottleneck: reserving d / 128 + 8 SMs, or 48, measured slower)
      const int cap = num_sms() - 24;
      e = syrk_tc(rest, aseg, bseg, 3, 128, C22, d, rows - LB, -1.f, 1.f, cap, st, cs->side);
      if (e == cudaErrorNotSupported)
        e = gemm_tc(rest, rest, 3, aseg, bseg, 128, C22, d, 0, rows - LB, rows - LB, -1.f, 1.f,
                    true, 1, st, cs->side);
      if (e != cudaSuccess) return e;
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
  return cholesky_inverse(L, Linv, d, T, sb, st, s);
}

}  // namespace ffh
