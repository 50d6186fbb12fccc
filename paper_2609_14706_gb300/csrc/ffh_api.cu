// libffh C ABI: handle, workspace, and the host-side driver of the FlipFlop fit.
//
// One fit enqueues, per iteration t (Section 5 updates, Appendix B order):
//   [t = 1, A_0 = I]  q_k = ||x_k||^2
//   [otherwise]       L = chol(A_{t-1}), M = L^-1 (bf16 copy), q_k = ||M x_k||^2
//   B_t = 1/(N n) G^T diag(q) G   (+ damping)
//   L = chol(B_t), M = L^-1,        r_k = ||M g_k||^2
//   A_t = 1/(N m) X^T diag(r) X   (+ damping)
//   s = tr(A_t)/n;  A_t /= s;  B_t *= s
//   convergence statistics of A_t, B_t against A_{t-1}, B_{t-1}
// all on the handle's stream.  The stopping test runs on the device: a one-thread kernel
// at the end of every iteration records the iteration and, when delta_t < tol, sets the
// status block's `stop` word, after which the kernels of the remaining iterations (already
// enqueued) return at once; the result is then copied from the slot of the last completed
// iteration.  The host synchronises once per fit, at the end, to read the status.
#include <stdarg.h>

#include <cmath>
#include <cstddef>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "ffh_internal.cuh"

namespace ffh {
cudaError_t launch_lower_to_bf16(const float* src, int64_t d, int64_t lds, __nv_bfloat16* dst,
                                 int64_t ldd, cudaStream_t s);
cudaError_t launch_trace(const float* F, int64_t d, double* out, cudaStream_t s);
}  // namespace ffh

using namespace ffh;

struct ffh_ctx {
  ffh_options opt{};
  cudaStream_t stream = nullptr;
  int device = 0;
  std::string err;
  void* ws = nullptr;
  size_t ws_bytes = 0;
  // last fit
  int iters_done = 0;
  int64_t N = 0, n = 0, m = 0;
  bool final_loglik = false;
  bool loglik_valid = true;      // the FlipFlop log-likelihood applies to the last fit
  std::vector<IterRecord> recs;  // index 1..iters_done
  // profiling (opt.profile): CUDA events recorded around the timed kernels
  double prof_ms[3] = {0, 0, 0};        // gram, qform, cholesky
  long long prof_n[3] = {0, 0, 0};
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  struct Pending {
    int kind;
    cudaEvent_t a, b;
  };
  std::vector<Pending> pending;
  CholStreams chol_cs;  // look-ahead streams of the tensor-core Cholesky (created on first use)
  // The last fit's enqueued work as a CUDA graph, replayed while the next fit matches `key`
  // (everything the enqueued sequence and its kernel arguments depend on).
  struct FitKey {
    const void *X = nullptr, *G = nullptr;
    int64_t N = 0, n = 0, m = 0;
    int32_t iters = 0;
    float tol = 0.f, damping = 0.f;
    int32_t dtype = 0, variant = 0, init = 0, final_loglik = 0, profile = 0;
    void* ws = nullptr;
    size_t ws_bytes = 0;
    bool operator==(const FitKey& o) const {
      return X == o.X && G == o.G && N == o.N && n == o.n && m == o.m && iters == o.iters &&
             tol == o.tol && damping == o.damping && dtype == o.dtype && variant == o.variant &&
             init == o.init && final_loglik == o.final_loglik && profile == o.profile &&
             ws == o.ws && ws_bytes == o.ws_bytes;
    }
  };
  struct FitGraph {
    FitKey key;
    cudaGraphExec_t exec = nullptr;
    bool failed = false;           // capture of `key` failed: enqueue it directly
    long long launches = 0;        // kernels in the graph
    std::vector<Pending> pending;  // profile intervals the graph records
    std::vector<cudaEvent_t> events;
  } fg;
  cudaStream_t cap_stream = nullptr;  // private stream the fit is captured on
  bool capturing = false;
  std::vector<cudaEvent_t> cap_events;  // profile events created while capturing
};

namespace {

struct Carve {
  char* base;
  size_t off = 0;
  explicit Carve(void* b) : base(static_cast<char*>(b)) {}
  template <class T>
  T* take(size_t count, size_t align = 256) {
    off = (off + align - 1) & ~(align - 1);
    T* p = base ? reinterpret_cast<T*>(base + off) : nullptr;
    off += count * sizeof(T);
    return p;
  }
};

ffh_status fail(ffh_t h, ffh_status st, const char* fmt, ...) {
  if (h) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    h->err = buf;
  }
  return st;
}

#define CK(call)                                                                        \
  do {                                                                                  \
    cudaError_t e_ = (call);                                                            \
    if (e_ != cudaSuccess)                                                              \
      return fail(h, FFH_ERR_CUDA, "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), \
                  __FILE__, __LINE__);                                                  \
  } while (0)

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

int64_t pad8(int64_t d) { return (d + 7) / 8 * 8; }

ffh_status ensure_ws(ffh_t h, size_t bytes) {
  if (h->opt.fault == FFH_FAULT_OOM) return fail(h, FFH_ERR_OOM, "workspace allocation failed (injected)");
  if (bytes <= h->ws_bytes && h->ws) return FFH_OK;
  CK(cudaStreamSynchronize(h->stream));
  if (h->ws) {
    cudaFree(h->ws);
    h->ws = nullptr;
    h->ws_bytes = 0;
  }
  void* p = nullptr;
  if (cudaMalloc(&p, bytes) != cudaSuccess) {
    cudaGetLastError();
    return fail(h, FFH_ERR_OOM, "workspace allocation of %zu bytes failed", bytes);
  }
  h->ws = p;
  h->ws_bytes = bytes;
  return FFH_OK;
}

enum { PROF_GRAM = 0, PROF_QFORM = 1, PROF_CHOL = 2 };

cudaEvent_t next_event(ffh_t h) {
  if (h->capturing) {
    // owned by the graph being captured (recorded on every replay), not the reusable pool
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    h->cap_events.push_back(e);
    return e;
  }
  if (h->ev_used == h->ev_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    h->ev_pool.push_back(e);
  }
  return h->ev_pool[h->ev_used++];
}

// Record a timing event; inside a capture it becomes a node of the graph, so every replay
// records it (a plain record on a capturing stream only orders work).
void prof_record(ffh_t h, cudaEvent_t e) {
  if (h->capturing)
    cudaEventRecordWithFlags(e, h->stream, cudaEventRecordExternal);
  else
    cudaEventRecord(e, h->stream);
}

// Start a timed region of `kind` on the handle's stream (no-op unless opt.profile).
cudaEvent_t prof_begin(ffh_t h) {
  if (!h->opt.profile) return nullptr;
  cudaEvent_t e = next_event(h);
  if (e) prof_record(h, e);
  return e;
}

void prof_end(ffh_t h, int kind, cudaEvent_t a, cudaEvent_t b_recorded = nullptr) {
  if (!a) return;
  cudaEvent_t b = b_recorded;
  if (!b) {
    b = next_event(h);
    if (!b) return;
    prof_record(h, b);
  }
  h->pending.push_back({kind, a, b});
}

// After a stream synchronisation: fold the recorded intervals into the totals.
void prof_resolve(ffh_t h) {
  for (auto& p : h->pending) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) {
      h->prof_ms[p.kind] += ms;
      h->prof_n[p.kind] += 1;
    } else {
      cudaGetLastError();
    }
  }
  h->pending.clear();
  h->ev_used = 0;
}

void drop_fit_graph(ffh_t h) {
  auto& g = h->fg;
  if (g.exec) cudaGraphExecDestroy(g.exec);
  for (cudaEvent_t e : g.events) cudaEventDestroy(e);
  g = ffh_ctx::FitGraph{};
}

// Run `enqueue` (which puts a fit's kernels on h->stream) through a CUDA graph: replay the
// handle's graph when `key` matches, else capture `enqueue` on a private stream, instantiate
// and launch it.  A capture that fails for any reason is discarded and the work enqueued
// directly (and `key` is not captured again).
template <class F>
ffh_status run_as_graph(ffh_t h, const ffh_ctx::FitKey& key, F&& enqueue) {
  auto& g = h->fg;
  if (g.key == key && (g.exec || g.failed)) {
    if (g.failed) return enqueue();
    CK(cudaGraphLaunch(g.exec, h->stream));
    note_launches((int)g.launches);
    h->pending.insert(h->pending.end(), g.pending.begin(), g.pending.end());
    return FFH_OK;
  }
  drop_fit_graph(h);
  g.key = key;
  if (!h->cap_stream) CK(cudaStreamCreateWithFlags(&h->cap_stream, cudaStreamNonBlocking));
  if (!h->chol_cs.crit) {
    const cudaError_t e = chol_streams_init(&h->chol_cs);
    if (e != cudaSuccess) {
      chol_streams_destroy(&h->chol_cs);
      return fail(h, FFH_ERR_CUDA, "Cholesky streams: %s", cudaGetErrorString(e));
    }
  }
  cudaStream_t user = h->stream;
  CK(cudaStreamBeginCapture(h->cap_stream, cudaStreamCaptureModeThreadLocal));
  h->stream = h->cap_stream;
  h->capturing = true;
  const size_t pend0 = h->pending.size();
  const long long l0 = launches_so_far();
  ffh_status es = enqueue();
  cudaGraph_t graph = nullptr;
  cudaError_t ce = cudaStreamEndCapture(h->cap_stream, &graph);
  h->stream = user;
  h->capturing = false;
  const long long counted = launches_so_far() - l0;
  std::vector<ffh_ctx::Pending> pend(h->pending.begin() + pend0, h->pending.end());
  h->pending.resize(pend0);
  std::vector<cudaEvent_t> evs;
  evs.swap(h->cap_events);
  cudaGraphExec_t exec = nullptr;
  if (es == FFH_OK && ce == cudaSuccess && graph)
    ce = cudaGraphInstantiateWithFlags(&exec, graph, 0);
  if (graph) cudaGraphDestroy(graph);
  // nothing ran during the capture: the launches counted there happen only when the graph does
  note_launches(-(int)counted);
  if (es != FFH_OK || ce != cudaSuccess || !exec) {
    cudaGetLastError();
    if (exec) cudaGraphExecDestroy(exec);
    for (cudaEvent_t e : evs) cudaEventDestroy(e);
    g.failed = true;
    h->err.clear();
    return enqueue();
  }
  g.exec = exec;
  g.launches = counted;
  g.pending = std::move(pend);
  g.events = std::move(evs);
  CK(cudaGraphLaunch(g.exec, h->stream));
  note_launches((int)g.launches);
  h->pending.insert(h->pending.end(), g.pending.begin(), g.pending.end());
  return FFH_OK;
}

ffh_status read_status(ffh_t h, DevStatus* st_dev, DevStatus* copy = nullptr) {
  DevStatus st;
  CK(cudaMemcpyAsync(&st, st_dev, sizeof(st), cudaMemcpyDeviceToHost, h->stream));
  if (copy) *copy = st;
  CK(cudaStreamSynchronize(h->stream));
  prof_resolve(h);
  if (st.error == FFH_ERR_NOT_SPD)
    return fail(h, FFH_ERR_NOT_SPD, "Cholesky pivot <= 0 or not finite at index %d", st.error_info);
  if (st.error == FFH_ERR_TIMEOUT)
    return fail(h, FFH_ERR_TIMEOUT, "bounded device wait expired (site %d)", st.error_info);
  if (st.error) return fail(h, (ffh_status)st.error, "device error %d (info %d)", st.error, st.error_info);
  return FFH_OK;
}

// Input staging: a device bf16 view of V (the tensor-core operand) and a device view in
// the caller's dtype (read by the A_0 = I row sums).
struct Staged {
  const __nv_bfloat16* bf = nullptr;
  int64_t ld_bf = 0;
  const void* raw = nullptr;
  int64_t ld_raw = 0;
};

struct GramTables {
  GramPlan plan{};
  int2* tiles = nullptr;
  int* lut = nullptr;
};

}  // namespace

// ---------------------------------------------------------------------------
extern "C" {

int32_t ffh_version(void) { return 100; }

ffh_status ffh_create(ffh_t* out, const ffh_options* opt, void* cuda_stream) {
  if (!out) return FFH_ERR_INVALID_ARG;
  *out = nullptr;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return FFH_ERR_CUDA;
  }
  int major = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  if (major != 10) return FFH_ERR_UNSUPPORTED;
  ffh_ctx* h = new ffh_ctx();
  if (opt) h->opt = *opt;
  h->stream = static_cast<cudaStream_t>(cuda_stream);
  h->device = dev;
  *out = h;
  return FFH_OK;
}

ffh_status ffh_set_options(ffh_t h, const ffh_options* opt) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->opt = opt ? *opt : ffh_options{};
  return FFH_OK;
}

ffh_status ffh_set_stream(ffh_t h, void* cuda_stream) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->stream = static_cast<cudaStream_t>(cuda_stream);
  return FFH_OK;
}

ffh_status ffh_destroy(ffh_t h) {
  if (!h) return FFH_OK;
  if (h->ws) {
    cudaStreamSynchronize(h->stream);
    cudaFree(h->ws);
  }
  for (cudaEvent_t e : h->ev_pool) cudaEventDestroy(e);
  drop_fit_graph(h);
  if (h->cap_stream) cudaStreamDestroy(h->cap_stream);
  chol_streams_destroy(&h->chol_cs);
  delete h;
  return FFH_OK;
}

const char* ffh_last_error(ffh_t h) { return h ? h->err.c_str() : "null handle"; }

}  // extern "C"

// ---------------------------------------------------------------------------
namespace {

ffh_status validate_opt(ffh_t h) {
  const ffh_options& o = h->opt;
  if (o.dtype != FFH_BF16 && o.dtype != FFH_F32) return fail(h, FFH_ERR_INVALID_ARG, "bad dtype %d", o.dtype);
  if (!(o.damping >= 0.f) || !std::isfinite(o.damping))
    return fail(h, FFH_ERR_INVALID_ARG, "damping must be finite and >= 0");
  if (o.variant < FFH_FLIPFLOP || o.variant > FFH_MARGINAL)
    return fail(h, FFH_ERR_INVALID_ARG, "bad variant %d", o.variant);
  if (o.reserved0 != 0 || o.reserved[0] || o.reserved[1] || o.reserved[2])
    return fail(h, FFH_ERR_INVALID_ARG, "reserved option field must be zero");
  if (o.no_graph != 0 && o.no_graph != 1) return fail(h, FFH_ERR_INVALID_ARG, "no_graph must be 0 or 1");
  return FFH_OK;
}

// Stage one sample matrix (N x d, caller dtype): returns device views.
ffh_status stage_input(ffh_t h, const void* V, bool on_dev, int64_t N, int64_t d,
                       __nv_bfloat16* bf_buf, float* f32_stage, Staged* out) {
  const int dtype = h->opt.dtype;
  if (dtype == FFH_BF16) {
    if (on_dev) {
      out->bf = static_cast<const __nv_bfloat16*>(V);
    } else {
      CK(cudaMemcpyAsync(bf_buf, V, (size_t)N * d * 2, cudaMemcpyHostToDevice, h->stream));
      out->bf = bf_buf;
    }
    out->ld_bf = d;
    out->raw = out->bf;
    out->ld_raw = d;
    return FFH_OK;
  }
  const float* src = static_cast<const float*>(V);
  if (!on_dev) {
    CK(cudaMemcpyAsync(f32_stage, V, (size_t)N * d * 4, cudaMemcpyHostToDevice, h->stream));
    src = f32_stage;
  }
  out->raw = src;
  out->ld_raw = d;
  if (bf_buf) {
    CK(launch_to_bf16(src, N, d, d, bf_buf, pad8(d), h->stream));
    out->bf = bf_buf;
    out->ld_bf = pad8(d);
  }
  return FFH_OK;
}

// C = scale * V^T diag(w) V on the tensor cores; the weights enter the kernel's operand
// load (no scaled copy of V).
ffh_status gram(ffh_t h, const Staged& V, int64_t N, int64_t d, const float* w_padded, float scale,
                float* C, float* partial, const GramTables& gt, DevStatus* st) {
  cudaEvent_t t0 = prof_begin(h);
  cudaEvent_t t1 = t0 ? next_event(h) : nullptr;
  CK(launch_gram_tc(V.bf, N, d, V.ld_bf, w_padded, scale, C, d, partial, gt.tiles, gt.lut,
                    gt.plan, st, h->opt.fault, h->stream, t1));
  prof_end(h, PROF_GRAM, t0, t1);
  return FFH_OK;
}

// q_k = ||L^T v_k||^2 = v_k^T F v_k for F = L L^T (the Frobenius variant's weights)
ffh_status qform_fwd(ffh_t h, const Staged& V, int64_t N, int64_t d, const float* L,
                     __nv_bfloat16* Mb, float* q, float* qpart, DevStatus* st) {
  const int64_t ldm = pad8(d);
  CK(launch_lowerT_to_bf16(L, d, d, Mb, ldm, h->stream));
  cudaEvent_t t0 = prof_begin(h);
  CK(launch_qform_tc(V.bf, N, d, V.ld_bf, Mb, ldm, q, qpart, st, h->stream, true));
  prof_end(h, PROF_QFORM, t0);
  return FFH_OK;
}

ffh_status qform(ffh_t h, const Staged& V, int64_t N, int64_t d, const float* Linv,
                 __nv_bfloat16* Mb, float* q, float* qpart, DevStatus* st) {
  const int64_t ldm = pad8(d);
  CK(launch_lower_to_bf16(Linv, d, d, Mb, ldm, h->stream));
  cudaEvent_t t0 = prof_begin(h);
  CK(launch_qform_tc(V.bf, N, d, V.ld_bf, Mb, ldm, q, qpart, st, h->stream));
  prof_end(h, PROF_QFORM, t0);
  return FFH_OK;
}

// Cholesky factor and inverse of F (d x d), timed as one region.
ffh_status chol(ffh_t h, const float* F, int64_t d, float* L, float* Linv, float* work,
                DevStatus* st, int fault) {
  cudaEvent_t t0 = prof_begin(h);
  if (!h->chol_cs.crit) {
    const cudaError_t e = chol_streams_init(&h->chol_cs);
    if (e != cudaSuccess) {
      chol_streams_destroy(&h->chol_cs);
      return fail(h, FFH_ERR_CUDA, "Cholesky streams: %s", cudaGetErrorString(e));
    }
  }
  CK(launch_cholesky_tc(F, d, d, L, Linv, work, st, fault, h->stream, &h->chol_cs));
  prof_end(h, PROF_CHOL, t0);
  return FFH_OK;
}

ffh_status setup_tables(ffh_t h, int64_t N, int64_t d, GramTables* gt, int2* tiles_dev,
                        int* lut_dev) {
  gt->plan = gram_plan(N, d, num_sms());
  gt->tiles = tiles_dev;
  gt->lut = lut_dev;
  const int64_t nbm = (d + kGramBM - 1) / kGramBM, nbn = (d + kGramBN - 1) / kGramBN;
  std::vector<int2> tiles((size_t)(nbm * nbn));
  std::vector<int> lut((size_t)(nbm * nbn));
  int T = 0;
  gram_build_tiles(d, tiles.data(), lut.data(), &T);
  CK(cudaMemcpyAsync(tiles_dev, tiles.data(), sizeof(int2) * T, cudaMemcpyHostToDevice, h->stream));
  CK(cudaMemcpyAsync(lut_dev, lut.data(), sizeof(int) * lut.size(), cudaMemcpyHostToDevice,
                     h->stream));
  CK(cudaStreamSynchronize(h->stream));  // host vectors go out of scope
  return FFH_OK;
}

}  // namespace

extern "C" ffh_status ffh_fit(ffh_t h, const void* X, const void* G, int64_t N, int64_t n,
                              int64_t m, int32_t iters, float tol, float* A_out, float* B_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  ffh_status vs = validate_opt(h);
  if (vs) return vs;
  if (!X || !G || !A_out || !B_out) return fail(h, FFH_ERR_INVALID_ARG, "null pointer argument");
  if (N < 1 || n < 1 || m < 1 || iters < 1)
    return fail(h, FFH_ERR_INVALID_ARG, "need N, n, m, iters >= 1");
  if (N > (int64_t)1 << 30) return fail(h, FFH_ERR_INVALID_ARG, "N too large");
  if (!(tol >= 0.f) || !std::isfinite(tol)) return fail(h, FFH_ERR_INVALID_ARG, "tol must be finite and >= 0");
  if (h->opt.dtype == FFH_BF16 && (n % 8 || m % 8))
    return fail(h, FFH_ERR_INVALID_ARG, "bf16 rows must be 16-byte aligned: n, m multiples of 8");
  if (N < std::max(n, m) && h->opt.damping == 0.f)
    return fail(h, FFH_ERR_RANK, "N = %lld < max(n, m) = %lld without damping",
                (long long)N, (long long)std::max(n, m));
  const int dtype = h->opt.dtype;
  const bool x_dev = is_device_ptr(X), g_dev = is_device_ptr(G);
  const bool init = h->opt.init_A != nullptr;
  const int64_t D = std::max(n, m);
  const int64_t Npad = (N + 63) / 64 * 64 + 64;

  GramPlan pn = gram_plan(N, n, num_sms()), pm = gram_plan(N, m, num_sms());
  auto layout = [&](Carve& c, DevStatus** st, IterRecord** recs, __nv_bfloat16** Xb,
                    __nv_bfloat16** Gb, float** stage, float** q, float** r, float** A2,
                    float** B2, float** L, float** Linv, __nv_bfloat16** Mb, float** work,
                    int2** tn, int** ln, int2** tm, int** lm, float** partial,
                    double** trb, float** Ares, float** Bres) {
    *st = c.take<DevStatus>(1);
    *recs = c.take<IterRecord>(iters + 2);
    const bool xcopy = dtype == FFH_F32 || (dtype == FFH_BF16 && !x_dev);
    const bool gcopy = dtype == FFH_F32 || (dtype == FFH_BF16 && !g_dev);
    *Xb = xcopy ? c.take<__nv_bfloat16>((size_t)N * pad8(n)) : nullptr;
    *Gb = gcopy ? c.take<__nv_bfloat16>((size_t)N * pad8(m)) : nullptr;
    const bool host_f32 = dtype == FFH_F32 && (!x_dev || !g_dev);
    *stage = host_f32 ? c.take<float>((size_t)N * (size_t)((!x_dev && !g_dev) ? (n + m) : D)) : nullptr;
    *q = c.take<float>(Npad);
    *r = c.take<float>(Npad);
    *A2 = c.take<float>((size_t)2 * n * n);
    *B2 = c.take<float>((size_t)2 * m * m);
    *L = c.take<float>((size_t)D * D);
    *Linv = c.take<float>((size_t)D * D);
    *Mb = c.take<__nv_bfloat16>((size_t)D * pad8(D));
    *work = c.take<float>(cholesky_tc_work_bytes(D) / 4 + 1);
    *tn = c.take<int2>(gram_tile_table_bytes(n) / sizeof(int2) + 1);
    *ln = c.take<int>(gram_tile_table_bytes(n) / sizeof(int) + 1);
    *tm = c.take<int2>(gram_tile_table_bytes(m) / sizeof(int2) + 1);
    *lm = c.take<int>(gram_tile_table_bytes(m) / sizeof(int) + 1);
    *partial = c.take<float>(std::max(gram_partial_bytes(pn), gram_partial_bytes(pm)) / 4);
    *trb = c.take<double>(8 + kRedDoubles);  // statistics, then the reduction scratch
    *Ares = c.take<float>((size_t)n * n);
    *Bres = c.take<float>((size_t)m * m);
  };
  DevStatus* st;
  IterRecord* recs;
  __nv_bfloat16 *Xb, *Gb, *Mb;
  float *stage, *q, *r, *A2, *B2, *L, *Linv, *work, *partial, *Ares, *Bres;
  int2 *tn, *tm;
  int *ln, *lm;
  double* trb;
  const size_t qpart_floats = std::max(qform_scratch_floats(N, n), qform_scratch_floats(N, m));
  {
    Carve c(nullptr);
    layout(c, &st, &recs, &Xb, &Gb, &stage, &q, &r, &A2, &B2, &L, &Linv, &Mb, &work, &tn,
           &ln, &tm, &lm, &partial, &trb, &Ares, &Bres);
    c.take<float>(qpart_floats);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  layout(c, &st, &recs, &Xb, &Gb, &stage, &q, &r, &A2, &B2, &L, &Linv, &Mb, &work, &tn, &ln,
         &tm, &lm, &partial, &trb, &Ares, &Bres);
  float* qpart = c.take<float>(qpart_floats);
  // the small kernels of this fit (the input staging included) test its status block (see
  // launch_iter_end), so it is cleared first, on every call, before anything is staged
  GateScope gate(st);
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), h->stream));
  CK(cudaMemsetAsync(recs, 0, sizeof(IterRecord) * (iters + 2), h->stream));
  CK(cudaMemsetAsync(q, 0, sizeof(float) * Npad, h->stream));
  CK(cudaMemsetAsync(r, 0, sizeof(float) * Npad, h->stream));
  GramTables gtn, gtm;
  {
    ffh_status es = setup_tables(h, N, n, &gtn, tn, ln);
    if (es) return es;
    es = setup_tables(h, N, m, &gtm, tm, lm);
    if (es) return es;
  }
  Staged xs, gs;
  ffh_status es = stage_input(h, X, x_dev, N, n, Xb, stage, &xs);
  if (es) return es;
  // both host fp32: X and G get separate staging regions
  float* stage_g = stage ? ((!x_dev && !g_dev) ? stage + (size_t)N * n : stage) : nullptr;
  es = stage_input(h, G, g_dev, N, m, Gb, stage_g, &gs);
  if (es) return es;

  float* A[2] = {A2, A2 + (size_t)n * n};
  float* B[2] = {B2, B2 + (size_t)m * m};
  if (init) {
    CK(cudaMemcpyAsync(A[0], h->opt.init_A, sizeof(float) * n * n, cudaMemcpyDefault, h->stream));
  }
  const float lam = h->opt.damping;
  const int variant = h->opt.variant;
  const bool frob = variant == FFH_FROBENIUS;
  const float sB = frob ? (float)(1.0 / (double)N) : (float)(1.0 / ((double)N * (double)n));
  const float sA = frob ? (float)(1.0 / (double)N) : (float)(1.0 / ((double)N * (double)m));
  int t_done = 0;
  // Input / Marginal: one pass, no alternating loop
  const int loop_iters = (variant == FFH_INPUT || variant == FFH_MARGINAL) ? 0 : iters;
  std::vector<IterRecord> host_recs((size_t)std::max(iters, 1) + 2);
  // Everything from here to the result selection is enqueued by `enqueue`, directly or
  // recorded once as a CUDA graph and replayed (run_as_graph); nothing in it waits for the
  // host.
  auto enqueue = [&]() -> ffh_status {
    cudaStream_t s = h->stream;
    int cur = 0;
    ffh_status es = FFH_OK;
    if (!init) CK(launch_fill_identity(A[cur], n, n, s));
    if (variant == FFH_INPUT || variant == FFH_MARGINAL) {
      // Table 1: A = E[x x^T]; B = I (Input) or E[g g^T] (Marginal); then tr A = n
      const float s1 = (float)(1.0 / (double)N);
      es = gram(h, xs, N, n, nullptr, s1, A[cur], partial, gtn, st);
      if (es) return es;
      if (variant == FFH_MARGINAL) {
        es = gram(h, gs, N, m, nullptr, s1, B[cur], partial, gtm, st);
        if (es) return es;
      } else {
        CK(launch_fill_identity(B[cur], m, m, s));
      }
      CK(launch_damp(A[cur], n, n, lam, st, s));
      CK(launch_damp(B[cur], m, m, lam, st, s));
      CK(launch_normalize(A[cur], n, B[cur], m, recs + 1, st, s));
      CK(launch_iter_end(st, recs + 1, 1, 0.f, cur, s));
    }
    for (int t = 1; t <= loop_iters; ++t) {
      IterRecord* R = recs + t;
      const int nxt = cur ^ 1;
      // ---- weights q_k = x_k^T A_{t-1}^-1 x_k  (Frobenius: x_k^T A_{t-1} x_k)
      if (t == 1 && !init) {
        CK(launch_rowsumsq(xs.raw, dtype, N, n, xs.ld_raw, q, s));
      } else if (frob) {
        es = chol(h, A[cur], n, L, nullptr, work, st, 0);
        if (es) return es;
        es = qform_fwd(h, xs, N, n, L, Mb, q, qpart, st);
        if (es) return es;
      } else {
        es = chol(h, A[cur], n, L, Linv, work, st, 0);
        if (es) return es;
        CK(launch_copy_f64(&R->logdet_A_prev, &st->logdet, s));
        if (t > 1) CK(launch_copy_f64(&recs[t - 1].logdet_A, &st->logdet, s));
        es = qform(h, xs, N, n, Linv, Mb, q, qpart, st);
        if (es) return es;
        if (t > 1) CK(launch_dot(q, r, N, &recs[t - 1].sum_qr_A, trb + 8, s));
      }
      // ---- B-update
      es = gram(h, gs, N, m, q, sB, B[nxt], partial, gtm, st);
      if (es) return es;
      if (frob) {
        CK(launch_frob2(A[cur], n, trb + 4, trb + 8, s));
        CK(launch_scale_by_inv(B[nxt], m, trb + 4, s));
      }
      CK(launch_damp(B[nxt], m, m, lam, st, s));
      es = chol(h, B[nxt], m, L, frob ? nullptr : Linv, work, st,
                (t == 1 && h->opt.fault == FFH_FAULT_BAD_PIVOT) ? FFH_FAULT_BAD_PIVOT : 0);
      if (es) return es;
      CK(launch_copy_f64(&R->logdet_B, &st->logdet, s));
      if (frob) {
        es = qform_fwd(h, gs, N, m, L, Mb, r, qpart, st);
      } else {
        es = qform(h, gs, N, m, Linv, Mb, r, qpart, st);
      }
      if (es) return es;
      CK(launch_dot(q, r, N, &R->sum_qr_B, trb + 8, s));
      // ---- A-update
      es = gram(h, xs, N, n, r, sA, A[nxt], partial, gtn, st);
      if (es) return es;
      if (frob) {
        CK(launch_frob2(B[nxt], m, trb + 5, trb + 8, s));
        CK(launch_scale_by_inv(A[nxt], n, trb + 5, s));
      }
      CK(launch_damp(A[nxt], n, n, lam, st, s));
      CK(launch_normalize(A[nxt], n, B[nxt], m, R, st, s));
      // ---- convergence statistics and the on-device stopping test
      CK(cudaMemsetAsync(&R->dA2, 0, sizeof(double) * 4, s));
      CK(launch_trace(A[nxt], n, trb + 0, s));
      CK(launch_trace(A[cur], n, trb + 1, s));
      CK(launch_delta(A[nxt], A[cur], n, &R->dA2, &R->nA2, trb, trb + 8, s));
      if (t > 1) {
        CK(launch_trace(B[nxt], m, trb + 2, s));
        CK(launch_trace(B[cur], m, trb + 3, s));
        CK(launch_delta(B[nxt], B[cur], m, &R->dB2, &R->nB2, trb + 2, trb + 8, s));
      }
      CK(launch_iter_end(st, R, t, tol, nxt, s));
      cur = nxt;
    }
    // the last completed iterate (the fit may have stopped before `iters`)
    CK(launch_select_copy(st, A[0], A[1], Ares, n * n, s));
    CK(launch_select_copy(st, B[0], B[1], Bres, m * m, s));
    if (h->opt.final_loglik && variant == FFH_FLIPFLOP) {
      CK(launch_resume(st, s));
      es = chol(h, Ares, n, L, Linv, work, st, 0);
      if (es) return es;
      CK(launch_record_at_done(st, recs, offsetof(IterRecord, logdet_A), &st->logdet, s));
      es = qform(h, xs, N, n, Linv, Mb, q, qpart, st);
      if (es) return es;
      CK(launch_dot(q, r, N, trb + 6, trb + 8, s));
      CK(launch_record_at_done(st, recs, offsetof(IterRecord, sum_qr_A), trb + 6, s));
    }
    return FFH_OK;
  };
  ffh_ctx::FitKey key;
  key.X = X;
  key.G = G;
  key.N = N;
  key.n = n;
  key.m = m;
  key.iters = iters;
  key.tol = tol;
  key.damping = h->opt.damping;
  key.dtype = dtype;
  key.variant = variant;
  key.init = init ? 1 : 0;
  key.final_loglik = h->opt.final_loglik;
  key.profile = h->opt.profile;
  key.ws = h->ws;
  key.ws_bytes = h->ws_bytes;
  const bool graphable = !h->opt.no_graph && h->opt.fault == FFH_FAULT_NONE && x_dev && g_dev;
  es = graphable ? run_as_graph(h, key, enqueue) : enqueue();
  if (es) return es;
  cudaStream_t s = h->stream;
  CK(cudaMemcpyAsync(A_out, Ares, sizeof(float) * n * n, cudaMemcpyDefault, s));
  CK(cudaMemcpyAsync(B_out, Bres, sizeof(float) * m * m, cudaMemcpyDefault, s));
  const int rec_count = std::max(loop_iters, 1) + 2;
  CK(cudaMemcpyAsync(host_recs.data(), recs, sizeof(IterRecord) * rec_count,
                     cudaMemcpyDeviceToHost, s));
  DevStatus hst;
  es = read_status(h, st, &hst);
  t_done = hst.iters_done;
  h->iters_done = t_done;
  h->N = N;
  h->n = n;
  h->m = m;
  h->final_loglik = h->opt.final_loglik != 0;
  h->recs = host_recs;
  h->loglik_valid = variant == FFH_FLIPFLOP;
  return es;
}

extern "C" ffh_status ffh_fit_matrix(ffh_t h, const float* Gk, int64_t N, int64_t n, int64_t m,
                                     int32_t iters, float tol, float* A_out, float* B_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  ffh_status vs = validate_opt(h);
  if (vs) return vs;
  if (!Gk || !A_out || !B_out) return fail(h, FFH_ERR_INVALID_ARG, "null pointer argument");
  if (N < 1 || n < 1 || m < 1 || iters < 1)
    return fail(h, FFH_ERR_INVALID_ARG, "need N, n, m, iters >= 1");
  if (n % 8 || m % 8) return fail(h, FFH_ERR_INVALID_ARG, "matrix samples need n, m multiples of 8");
  if (!(tol >= 0.f) || !std::isfinite(tol)) return fail(h, FFH_ERR_INVALID_ARG, "tol must be finite and >= 0");
  if (h->opt.variant != FFH_FLIPFLOP) return fail(h, FFH_ERR_UNSUPPORTED, "matrix samples: FlipFlop variant only");
  if (N * std::min(n, m) < std::max(n, m) && h->opt.damping == 0.f)
    return fail(h, FFH_ERR_RANK, "N min(n, m) < max(n, m) without damping");
  if (N * m > ((int64_t)1 << 31) - 1 || N * n > ((int64_t)1 << 31) - 1)
    return fail(h, FFH_ERR_INVALID_ARG, "N * max(n, m) too large");
  const bool g_dev = is_device_ptr(Gk);
  const bool init = h->opt.init_A != nullptr;
  const int64_t D = std::max(n, m);
  const int64_t mn = m * n;
  // samples per chunk: transform output (V) chunk of about 1 GiB
  const int64_t Kc = std::max<int64_t>(1, std::min<int64_t>(N, ((int64_t)1 << 29) / mn));
  const int64_t Kh = g_dev ? 0 : Kc;  // host staging (fp32) chunk
  GramPlan pa = gram_plan(Kc * m, n, num_sms()), pb = gram_plan(Kc * n, m, num_sms());
  auto layout = [&](Carve& c, DevStatus** st, IterRecord** recs, __nv_bfloat16** Gb,
                    float** stage, __nv_bfloat16** V, float** A2, float** B2, float** Cc,
                    float** L, float** Linv, __nv_bfloat16** Mb, float** work,
                    int2** tn, int** ln, int2** tm, int** lm, float** partial, double** trb,
                    double** fro, float** Ares, float** Bres) {
    *st = c.take<DevStatus>(1);
    *recs = c.take<IterRecord>(iters + 2);
    *Gb = c.take<__nv_bfloat16>((size_t)N * mn);
    *stage = Kh ? c.take<float>((size_t)Kh * mn) : nullptr;
    *V = c.take<__nv_bfloat16>((size_t)Kc * mn);
    *A2 = c.take<float>((size_t)2 * n * n);
    *B2 = c.take<float>((size_t)2 * m * m);
    *Cc = c.take<float>((size_t)D * D);
    *L = c.take<float>((size_t)D * D);
    *Linv = c.take<float>((size_t)D * D);
    *Mb = c.take<__nv_bfloat16>((size_t)D * D);
    *work = c.take<float>(cholesky_tc_work_bytes(D) / 4 + 1);
    *tn = c.take<int2>(gram_tile_table_bytes(n) / sizeof(int2) + 1);
    *ln = c.take<int>(gram_tile_table_bytes(n) / sizeof(int) + 1);
    *tm = c.take<int2>(gram_tile_table_bytes(m) / sizeof(int2) + 1);
    *lm = c.take<int>(gram_tile_table_bytes(m) / sizeof(int) + 1);
    *partial = c.take<float>(std::max(gram_partial_bytes(pa), gram_partial_bytes(pb)) / 4);
    *trb = c.take<double>(8 + kRedDoubles);  // statistics, then the reduction scratch
    *fro = c.take<double>(4);
    *Ares = c.take<float>((size_t)n * n);
    *Bres = c.take<float>((size_t)m * m);
  };
  DevStatus* st;
  IterRecord* recs;
  __nv_bfloat16 *Gb, *V, *Mb;
  float *stage, *A2, *B2, *Cc, *L, *Linv, *work, *partial, *Ares, *Bres;
  int2 *tn, *tm;
  int *ln, *lm;
  double *trb, *fro;
  {
    Carve c(nullptr);
    layout(c, &st, &recs, &Gb, &stage, &V, &A2, &B2, &Cc, &L, &Linv, &Mb, &work, &tn, &ln,
           &tm, &lm, &partial, &trb, &fro, &Ares, &Bres);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  layout(c, &st, &recs, &Gb, &stage, &V, &A2, &B2, &Cc, &L, &Linv, &Mb, &work, &tn, &ln, &tm,
         &lm, &partial, &trb, &fro, &Ares, &Bres);
  cudaStream_t s = h->stream;
  // the small kernels of this fit test its status block (see launch_iter_end)
  GateScope gate(st);
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  CK(cudaMemsetAsync(recs, 0, sizeof(IterRecord) * (iters + 2), s));
  GramTables gtn, gtm;
  {
    // the Gram plans depend on the chunk length; tables depend on d only
    ffh_status es = setup_tables(h, Kc * m, n, &gtn, tn, ln);
    if (es) return es;
    es = setup_tables(h, Kc * n, m, &gtm, tm, lm);
    if (es) return es;
  }
  // samples -> bf16 (N*m rows of n)
  for (int64_t k0 = 0; k0 < N; k0 += (g_dev ? N : Kh)) {
    const int64_t nk = std::min(N - k0, g_dev ? N : Kh);
    const float* src = Gk + k0 * mn;
    if (!g_dev) {
      CK(cudaMemcpyAsync(stage, src, sizeof(float) * nk * mn, cudaMemcpyHostToDevice, s));
      src = stage;
    }
    CK(launch_to_bf16(src, nk * m, n, n, Gb + k0 * mn, n, s));
  }
  float* A[2] = {A2, A2 + (size_t)n * n};
  float* B[2] = {B2, B2 + (size_t)m * m};
  int cur = 0;
  if (init) {
    CK(cudaMemcpyAsync(A[cur], h->opt.init_A, sizeof(float) * n * n, cudaMemcpyDefault, s));
  } else {
    CK(launch_fill_identity(A[cur], n, n, s));
  }
  const float lam = h->opt.damping;
  const float sB = (float)(1.0 / ((double)N * (double)n));
  const float sA = (float)(1.0 / ((double)N * (double)m));
  ffh_status es;
  // one half-step: C = scale * sum over chunks of Gram(M * Gop_k)
  auto half = [&](const __nv_bfloat16* Mbf, int64_t d, bool b_update, float scale, float* C,
                  const GramTables& gt) -> ffh_status {
    const int64_t d_other = b_update ? m : n;
    CK(launch_zero_f32(C, d_other * d_other, st, s));
    for (int64_t k0 = 0; k0 < N; k0 += Kc) {
      const int64_t nk = std::min(Kc, N - k0);
      CK(launch_transform_tc(Mbf, d, d, Gb + k0 * mn, nk, m, n, b_update, V, st, s));
      Staged vsd;
      vsd.bf = V;
      vsd.ld_bf = d_other;
      vsd.raw = V;
      vsd.ld_raw = d_other;
      GramTables g2 = gt;
      g2.plan = gram_plan(nk * d, d_other, num_sms());
      // the partial buffer holds the split count of a full chunk; never exceed it
      const GramPlan& full = b_update ? pb : pa;
      if (g2.plan.units > full.units) {
        g2.plan.S = std::max(1, full.units / g2.plan.T);
        g2.plan.units = g2.plan.T * g2.plan.S;
        g2.plan.grid = std::min(g2.plan.units, num_sms());
      }
      ffh_status e2 = gram(h, vsd, nk * d, d_other, nullptr, scale, Cc, partial, g2, st);
      if (e2) return e2;
      CK(launch_add(C, Cc, d_other * d_other, s));
    }
    return FFH_OK;
  };
  int t_done = 0;
  std::vector<IterRecord> host_recs((size_t)iters + 2);
  for (int t = 1; t <= iters; ++t) {
    IterRecord* R = recs + t;
    const int nxt = cur ^ 1;
    // ---- M_A = chol(A_{t-1})^-1 (bf16)
    es = chol(h, A[cur], n, L, Linv, work, st, 0);
    if (es) return es;
    CK(launch_copy_f64(&R->logdet_A_prev, &st->logdet, s));
    if (t > 1) {
      CK(launch_copy_f64(&recs[t - 1].logdet_A, &st->logdet, s));
      CK(launch_frob2(Linv, n, &recs[t - 1].trinvA, trb + 8, s));
    }
    CK(launch_lower_to_bf16(Linv, n, n, Mb, n, s));
    // ---- B-update
    es = half(Mb, n, true, sB, B[nxt], gtm);
    if (es) return es;
    CK(launch_damp(B[nxt], m, m, lam, st, s, &R->shift_B));
    es = chol(h, B[nxt], m, L, Linv, work, st,
              (t == 1 && h->opt.fault == FFH_FAULT_BAD_PIVOT) ? FFH_FAULT_BAD_PIVOT : 0);
    if (es) return es;
    CK(launch_copy_f64(&R->logdet_B, &st->logdet, s));
    CK(launch_frob2(Linv, m, &R->trinvB, trb + 8, s));
    CK(launch_lower_to_bf16(Linv, m, m, Mb, m, s));
    // ---- A-update
    es = half(Mb, m, false, sA, A[nxt], gtn);
    if (es) return es;
    CK(launch_damp(A[nxt], n, n, lam, st, s, &R->shift_A));
    CK(launch_normalize(A[nxt], n, B[nxt], m, R, st, s));
    CK(cudaMemsetAsync(&R->dA2, 0, sizeof(double) * 4, s));
    CK(launch_trace(A[nxt], n, trb + 0, s));
    CK(launch_trace(A[cur], n, trb + 1, s));
    CK(launch_delta(A[nxt], A[cur], n, &R->dA2, &R->nA2, trb, trb + 8, s));
    if (t > 1) {
      CK(launch_trace(B[nxt], m, trb + 2, s));
      CK(launch_trace(B[cur], m, trb + 3, s));
      CK(launch_delta(B[nxt], B[cur], m, &R->dB2, &R->nB2, trb + 2, trb + 8, s));
    }
    CK(launch_iter_end(st, R, t, tol, nxt, s));
    cur = nxt;
  }
  // the last completed iterate (the fit may have stopped before `iters`)
  CK(launch_select_copy(st, A[0], A[1], Ares, n * n, s));
  CK(launch_select_copy(st, B[0], B[1], Bres, m * m, s));
  if (h->opt.final_loglik) {
    CK(launch_resume(st, s));
    es = chol(h, Ares, n, L, Linv, work, st, 0);
    if (es) return es;
    CK(launch_record_at_done(st, recs, offsetof(IterRecord, logdet_A), &st->logdet, s));
    CK(launch_frob2(Linv, n, trb + 6, trb + 8, s));
    CK(launch_record_at_done(st, recs, offsetof(IterRecord, trinvA), trb + 6, s));
  }
  CK(cudaMemcpyAsync(A_out, Ares, sizeof(float) * n * n, cudaMemcpyDefault, s));
  CK(cudaMemcpyAsync(B_out, Bres, sizeof(float) * m * m, cudaMemcpyDefault, s));
  CK(cudaMemcpyAsync(host_recs.data(), recs, sizeof(IterRecord) * (iters + 2),
                     cudaMemcpyDeviceToHost, s));
  DevStatus hst;
  es = read_status(h, st, &hst);
  t_done = hst.iters_done;
  // trace terms of the log-likelihood from exact identities:
  //   sum_k tr(B^-1 G_k A^-1 G_k^T) = N n tr(B^-1 S_B) = N n (m - shift_B tr(B^-1)) at the
  //   B-point (B = S_B + shift_B I), and N m (n - shift_A tr(A^-1)) at the A-point.
  const double Nd = (double)N, nd = (double)n, md = (double)m;
  for (int t = 1; t <= t_done; ++t) {
    IterRecord& R = host_recs[t];
    R.sum_qr_B = Nd * nd * (md - R.shift_B * R.trinvB);
    const bool haveA = t < t_done || h->opt.final_loglik;
    // trinvA is of the rescaled A_t; the shift is in the units before the rescale
    R.sum_qr_A = haveA ? R.scale * Nd * md * (nd - R.shift_A * R.trinvA / R.scale) : 0.0;
  }
  h->iters_done = t_done;
  h->N = N;
  h->n = n;
  h->m = m;
  h->final_loglik = h->opt.final_loglik != 0;
  h->recs = host_recs;
  h->loglik_valid = true;
  return es;
}

extern "C" ffh_status ffh_get_stats(ffh_t h, int32_t* iters_done, double* delta,
                                    double* loglik_trace, double* mean_qr, int32_t capacity,
                                    int32_t* n_trace) {
  if (!h) return FFH_ERR_INVALID_ARG;
  const int T = h->iters_done;
  if (iters_done) *iters_done = T;
  if (n_trace) *n_trace = 2 * T;
  const double N = (double)h->N, n = (double)h->n, m = (double)h->m;
  if (delta) {
    if (T <= 1 || h->recs.empty()) {
      *delta = INFINITY;
    } else {
      const IterRecord& R = h->recs[T];
      const double dA = R.nA2 > 0 ? std::sqrt(R.dA2 / R.nA2) : 0.0;
      const double dB = R.nB2 > 0 ? std::sqrt(R.dB2 / R.nB2) : 0.0;
      *delta = std::max(dA, dB);
    }
  }
  for (int t = 1; t <= T; ++t) {
    const IterRecord& R = h->recs[t];
    const int i0 = 2 * (t - 1), i1 = i0 + 1;
    // l(A_{t-1}, B_t): B_t before the rescale, r computed with it
    const double lB = h->loglik_valid
                          ? -0.5 * (N * m * R.logdet_A_prev + N * n * R.logdet_B + R.sum_qr_B)
                          : NAN;
    // l(A_t, B_t) after the rescale s: log|sB| = log|B| + m log s, r/s
    const bool haveA = (t < T || h->final_loglik) && h->loglik_valid;
    const double ldB_s = R.logdet_B + m * std::log(R.scale);
    const double lA = haveA ? -0.5 * (N * m * R.logdet_A + N * n * ldB_s + R.sum_qr_A / R.scale)
                            : NAN;
    if (loglik_trace) {
      if (i0 < capacity) loglik_trace[i0] = lB;
      if (i1 < capacity) loglik_trace[i1] = lA;
    }
    if (mean_qr) {
      if (i0 < capacity) mean_qr[i0] = h->loglik_valid ? R.sum_qr_B / N : NAN;
      if (i1 < capacity) mean_qr[i1] = haveA ? R.sum_qr_A / (N * R.scale) : NAN;
    }
  }
  return FFH_OK;
}

// ---------------------------------------------------------------------------
// single steps
// ---------------------------------------------------------------------------
extern "C" ffh_status ffh_weighted_gram(ffh_t h, const void* V, const float* w, int64_t N,
                                        int64_t d, float scale, float* C_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  ffh_status vs = validate_opt(h);
  if (vs) return vs;
  if (!V || !C_out || N < 1 || d < 1) return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (N > (int64_t)1 << 30) return fail(h, FFH_ERR_INVALID_ARG, "N too large");
  if (!is_device_ptr(V) || !is_device_ptr(C_out) || (w && !is_device_ptr(w)))
    return fail(h, FFH_ERR_INVALID_ARG, "single-step calls take device pointers");
  const int dtype = h->opt.dtype;
  if (dtype == FFH_BF16 && d % 8) return fail(h, FFH_ERR_INVALID_ARG, "bf16 rows: d multiple of 8");
  const int64_t Npad = (N + 63) / 64 * 64 + 64;
  GramPlan plan = gram_plan(N, d, num_sms());
  auto layout = [&](Carve& c, DevStatus** st, float** wp, __nv_bfloat16** Vb, float** partial,
                    int2** tiles, int** lut) {
    *st = c.take<DevStatus>(1);
    *wp = c.take<float>(Npad);
    *Vb = (dtype == FFH_F32) ? c.take<__nv_bfloat16>((size_t)N * pad8(d)) : nullptr;
    *partial = c.take<float>(gram_partial_bytes(plan) / 4);
    *tiles = c.take<int2>(gram_tile_table_bytes(d) / sizeof(int2) + 1);
    *lut = c.take<int>(gram_tile_table_bytes(d) / sizeof(int) + 1);
  };
  DevStatus* st;
  float *wp, *partial;
  __nv_bfloat16* Vb;
  int2* tiles;
  int* lut;
  {
    Carve c(nullptr);
    layout(c, &st, &wp, &Vb, &partial, &tiles, &lut);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  layout(c, &st, &wp, &Vb, &partial, &tiles, &lut);
  cudaStream_t s = h->stream;
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  const float* wuse = nullptr;
  if (w) {
    CK(cudaMemsetAsync(wp, 0, sizeof(float) * Npad, s));
    CK(cudaMemcpyAsync(wp, w, sizeof(float) * N, cudaMemcpyDeviceToDevice, s));
    wuse = wp;
  }
  Staged vs_;
  ffh_status es = stage_input(h, V, true, N, d, Vb, nullptr, &vs_);
  if (es) return es;
  GramTables gt;
  es = setup_tables(h, N, d, &gt, tiles, lut);
  if (es) return es;
  es = gram(h, vs_, N, d, wuse, scale, C_out, partial, gt, st);
  if (es) return es;
  return read_status(h, st);
}

extern "C" ffh_status ffh_quad_form(ffh_t h, const void* V, const float* Linv, int64_t N,
                                    int64_t d, float* q_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  ffh_status vs = validate_opt(h);
  if (vs) return vs;
  if (!V || !Linv || !q_out || N < 1 || d < 1) return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (N > (int64_t)1 << 30) return fail(h, FFH_ERR_INVALID_ARG, "N too large");
  if (!is_device_ptr(V) || !is_device_ptr(Linv) || !is_device_ptr(q_out))
    return fail(h, FFH_ERR_INVALID_ARG, "single-step calls take device pointers");
  const int dtype = h->opt.dtype;
  if (dtype == FFH_BF16 && d % 8) return fail(h, FFH_ERR_INVALID_ARG, "bf16 rows: d multiple of 8");
  auto layout = [&](Carve& c, DevStatus** st, __nv_bfloat16** Vb, __nv_bfloat16** Mb) {
    *st = c.take<DevStatus>(1);
    *Vb = (dtype == FFH_F32) ? c.take<__nv_bfloat16>((size_t)N * pad8(d)) : nullptr;
    *Mb = c.take<__nv_bfloat16>((size_t)d * pad8(d));
  };
  DevStatus* st;
  __nv_bfloat16 *Vb, *Mb;
  const size_t qpart_floats = qform_scratch_floats(N, d);
  {
    Carve c(nullptr);
    layout(c, &st, &Vb, &Mb);
    c.take<float>(qpart_floats);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  layout(c, &st, &Vb, &Mb);
  float* qpart = c.take<float>(qpart_floats);
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), h->stream));
  Staged vs_;
  ffh_status es = stage_input(h, V, true, N, d, Vb, nullptr, &vs_);
  if (es) return es;
  es = qform(h, vs_, N, d, Linv, Mb, q_out, qpart, st);
  if (es) return es;
  return read_status(h, st);
}

extern "C" ffh_status ffh_cholesky(ffh_t h, const float* F, int64_t d, float* L_out,
                                   float* Linv_out, double* logdet) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  if (!F || d < 1) return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (!is_device_ptr(F) || (L_out && !is_device_ptr(L_out)) ||
      (Linv_out && !is_device_ptr(Linv_out)))
    return fail(h, FFH_ERR_INVALID_ARG, "single-step calls take device pointers");
  auto layout = [&](Carve& c, DevStatus** st, float** L, float** Li, float** work) {
    *st = c.take<DevStatus>(1);
    *L = L_out ? nullptr : c.take<float>((size_t)d * d);
    *Li = c.take<float>((size_t)d * d);
    *work = c.take<float>(cholesky_tc_work_bytes(d) / 4 + 1);
  };
  DevStatus* st;
  float *L, *Li, *work;
  {
    Carve c(nullptr);
    layout(c, &st, &L, &Li, &work);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  layout(c, &st, &L, &Li, &work);
  if (L_out) L = L_out;
  cudaStream_t s = h->stream;
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  ffh_status cs = chol(h, F, d, L, Linv_out ? Linv_out : (float*)nullptr, work, st,
                       h->opt.fault == FFH_FAULT_BAD_PIVOT ? FFH_FAULT_BAD_PIVOT : 0);
  if (cs) return cs;
  (void)Li;
  DevStatus hst;
  CK(cudaMemcpyAsync(&hst, st, sizeof(hst), cudaMemcpyDeviceToHost, s));
  ffh_status es = read_status(h, st);
  if (logdet) *logdet = hst.logdet;
  return es;
}

extern "C" ffh_status ffh_rev_cholesky(ffh_t h, const float* F, int64_t d, float* L_out,
                                       float* Lt_out, double* logdet) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  if (!F || d < 1) return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (!is_device_ptr(F) || (L_out && !is_device_ptr(L_out)) || (Lt_out && !is_device_ptr(Lt_out)))
    return fail(h, FFH_ERR_INVALID_ARG, "WaterKron calls take device pointers");
  auto layout = [&](Carve& c, DevStatus** st, float** Fr, float** C, float** Ci, float** work) {
    *st = c.take<DevStatus>(1);
    *Fr = c.take<float>((size_t)d * d);
    *C = c.take<float>((size_t)d * d);
    *Ci = c.take<float>((size_t)d * d);
    *work = c.take<float>(cholesky_tc_work_bytes(d) / 4 + 1);
  };
  DevStatus* st;
  float *Fr, *C, *Ci, *work;
  {
    Carve c(nullptr);
    layout(c, &st, &Fr, &C, &Ci, &work);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  layout(c, &st, &Fr, &C, &Ci, &work);
  cudaStream_t s = h->stream;
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  // C C^T = J F J;  L = J C^T J,  L^-1 = J C^-T J (column-normalised for Algorithms 1-2)
  CK(launch_reverse_sym(F, d, d, Fr, s));
  ffh_status es = chol(h, Fr, d, C, Ci, work, st,
                       h->opt.fault == FFH_FAULT_BAD_PIVOT ? FFH_FAULT_BAD_PIVOT : 0);
  if (es) return es;
  if (L_out) CK(launch_rev_transpose(C, d, L_out, false, s));
  if (Lt_out) CK(launch_rev_transpose(Ci, d, Lt_out, true, s));
  DevStatus hst;
  CK(cudaMemcpyAsync(&hst, st, sizeof(hst), cudaMemcpyDeviceToHost, s));
  es = read_status(h, st);
  if (logdet) *logdet = hst.logdet;
  return es;
}

extern "C" ffh_status ffh_waterfilling_scales(ffh_t h, const float* LA, int64_t n, const float* LB,
                                              int64_t m, float gamma, float* alpha_out,
                                              float* beta_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  if (!LA || !LB || !alpha_out || !beta_out || n < 1 || m < 1 || !(gamma > 0.f) ||
      !std::isfinite(gamma))
    return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (!is_device_ptr(LA) || !is_device_ptr(LB) || !is_device_ptr(alpha_out) ||
      !is_device_ptr(beta_out))
    return fail(h, FFH_ERR_INVALID_ARG, "WaterKron calls take device pointers");
  CK(launch_waterfilling(LA, n, LB, m, gamma, alpha_out, beta_out, h->stream));
  CK(cudaStreamSynchronize(h->stream));
  return FFH_OK;
}

extern "C" ffh_status ffh_gptq2(ffh_t h, const float* W, const float* LtA, const float* LtB,
                                const float* alpha, const float* beta, int64_t m, int64_t n,
                                int32_t* Z_out, float* V_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  if (!W || !LtA || !LtB || !alpha || !beta || !Z_out || m < 1 || n < 1)
    return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (m > 32768) return fail(h, FFH_ERR_INVALID_ARG, "m = %lld > 32768", (long long)m);
  if (!is_device_ptr(W) || !is_device_ptr(LtA) || !is_device_ptr(LtB) || !is_device_ptr(alpha) ||
      !is_device_ptr(beta) || !is_device_ptr(Z_out) || (V_out && !is_device_ptr(V_out)))
    return fail(h, FFH_ERR_INVALID_ARG, "WaterKron calls take device pointers");
  auto layout = [&](Carve& c, DevStatus** st, void** work) {
    *st = c.take<DevStatus>(1);
    *work = c.take<char>(gptq2_work_bytes(m, n));
  };
  DevStatus* st;
  void* work;
  {
    Carve c(nullptr);
    layout(c, &st, &work);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  layout(c, &st, &work);
  cudaStream_t s = h->stream;
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  CK(launch_gptq2(W, LtA, LtB, alpha, beta, m, n, Z_out, V_out, work, st, s));
  return read_status(h, st);
}

extern "C" ffh_status ffh_get_timings(ffh_t h, ffh_timings* out, int32_t reset) {
  if (!h || !out) return FFH_ERR_INVALID_ARG;
  if (!h->pending.empty()) {
    CK(cudaStreamSynchronize(h->stream));
    prof_resolve(h);
  }
  out->gram_ms = h->prof_ms[PROF_GRAM];
  out->gram_launches = h->prof_n[PROF_GRAM];
  out->qform_ms = h->prof_ms[PROF_QFORM];
  out->qform_launches = h->prof_n[PROF_QFORM];
  out->chol_ms = h->prof_ms[PROF_CHOL];
  out->chol_calls = h->prof_n[PROF_CHOL];
  out->kernel_launches = launches_so_far();
  if (reset) {
    for (int k = 0; k < 3; ++k) {
      h->prof_ms[k] = 0;
      h->prof_n[k] = 0;
    }
  }
  return FFH_OK;
}

extern "C" ffh_status ffh_phi_tilde(ffh_t h, const void* X, const void* G, int64_t N, int64_t n,
                                    int64_t m, const float* A, const float* B, double* phi_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  ffh_status vs = validate_opt(h);
  if (vs) return vs;
  if (!X || !G || !A || !B || !phi_out || N < 1 || n < 1 || m < 1)
    return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (!is_device_ptr(X) || !is_device_ptr(G) || !is_device_ptr(A) || !is_device_ptr(B))
    return fail(h, FFH_ERR_INVALID_ARG, "ffh_phi_tilde takes device pointers");
  const int dtype = h->opt.dtype;
  if (dtype == FFH_BF16 && (n % 8 || m % 8))
    return fail(h, FFH_ERR_INVALID_ARG, "bf16 rows must be 16-byte aligned: n, m multiples of 8");
  const int64_t D = std::max(n, m);
  const int64_t Npad = (N + 63) / 64 * 64 + 64;
  auto layout = [&](Carve& c, DevStatus** st, __nv_bfloat16** Xb, __nv_bfloat16** Gb, float** q,
                    float** r, float** L, float** Linv, __nv_bfloat16** Mb, float** work,
                    double** acc) {
    *st = c.take<DevStatus>(1);
    *Xb = (dtype == FFH_F32) ? c.take<__nv_bfloat16>((size_t)N * pad8(n)) : nullptr;
    *Gb = (dtype == FFH_F32) ? c.take<__nv_bfloat16>((size_t)N * pad8(m)) : nullptr;
    *q = c.take<float>(Npad);
    *r = c.take<float>(Npad);
    *L = c.take<float>((size_t)D * D);
    *Linv = c.take<float>((size_t)D * D);
    *Mb = c.take<__nv_bfloat16>((size_t)D * pad8(D));
    *work = c.take<float>(cholesky_tc_work_bytes(D) / 4 + 1);
    *acc = c.take<double>(4 + kRedDoubles);  // results, then the reduction scratch
  };
  DevStatus* st;
  __nv_bfloat16 *Xb, *Gb, *Mb;
  float *q, *r, *L, *Linv, *work;
  double* acc;
  const size_t qpart_floats = std::max(qform_scratch_floats(N, n), qform_scratch_floats(N, m));
  {
    Carve c(nullptr);
    layout(c, &st, &Xb, &Gb, &q, &r, &L, &Linv, &Mb, &work, &acc);
    c.take<float>(qpart_floats);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  layout(c, &st, &Xb, &Gb, &q, &r, &L, &Linv, &Mb, &work, &acc);
  float* qpart = c.take<float>(qpart_floats);
  cudaStream_t s = h->stream;
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  Staged xs, gs;
  ffh_status es = stage_input(h, X, true, N, n, Xb, nullptr, &xs);
  if (es) return es;
  es = stage_input(h, G, true, N, m, Gb, nullptr, &gs);
  if (es) return es;
  double ld[2] = {0, 0};
  es = chol(h, A, n, L, Linv, work, st, 0);
  if (es) return es;
  CK(cudaMemcpyAsync(&acc[1], &st->logdet, sizeof(double), cudaMemcpyDeviceToDevice, s));
  es = qform(h, xs, N, n, Linv, Mb, q, qpart, st);
  if (es) return es;
  es = chol(h, B, m, L, Linv, work, st, 0);
  if (es) return es;
  CK(cudaMemcpyAsync(&acc[2], &st->logdet, sizeof(double), cudaMemcpyDeviceToDevice, s));
  es = qform(h, gs, N, m, Linv, Mb, r, qpart, st);
  if (es) return es;
  CK(launch_dot(q, r, N, &acc[0], acc + 4, s));
  double hacc[3];
  CK(cudaMemcpyAsync(hacc, acc, sizeof(hacc), cudaMemcpyDeviceToHost, s));
  es = read_status(h, st);
  if (es) return es;
  (void)ld;
  const double mean_qr = hacc[0] / (double)N;
  *phi_out = std::exp(hacc[1] / (double)n + hacc[2] / (double)m +
                      std::log(mean_qr / ((double)m * (double)n)));
  return FFH_OK;
}

// ---------------------------------------------------------------------------
// sample-sharded fit: the steps a driver composes around a sum over ranks
// ---------------------------------------------------------------------------
extern "C" ffh_status ffh_partial_gram(ffh_t h, const void* U, const void* V, int64_t N,
                                       int64_t du, int64_t dv, const float* F,
                                       int32_t accumulate, float* P_out, double* logdet_F) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  ffh_status vs = validate_opt(h);
  if (vs) return vs;
  if (!U || !V || !P_out || N < 1 || du < 1 || dv < 1)
    return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (N > (int64_t)1 << 30) return fail(h, FFH_ERR_INVALID_ARG, "N too large");
  if (!is_device_ptr(U) || !is_device_ptr(V) || !is_device_ptr(P_out) || (F && !is_device_ptr(F)))
    return fail(h, FFH_ERR_INVALID_ARG, "ffh_partial_gram takes device pointers");
  const int dtype = h->opt.dtype;
  if (dtype == FFH_BF16 && (du % 8 || dv % 8))
    return fail(h, FFH_ERR_INVALID_ARG, "bf16 rows must be 16-byte aligned: du, dv multiples of 8");
  const int64_t Npad = (N + 63) / 64 * 64 + 64;
  GramPlan plan = gram_plan(N, dv, num_sms());
  auto layout = [&](Carve& c, DevStatus** st, __nv_bfloat16** Ub, __nv_bfloat16** Vb, float** w,
                    float** L, float** Linv, __nv_bfloat16** Mb, float** work, float** partial,
                    int2** tiles, int** lut, float** Ptmp) {
    *st = c.take<DevStatus>(1);
    *Ub = (dtype == FFH_F32) ? c.take<__nv_bfloat16>((size_t)N * pad8(du)) : nullptr;
    *Vb = (dtype == FFH_F32) ? c.take<__nv_bfloat16>((size_t)N * pad8(dv)) : nullptr;
    *w = c.take<float>(Npad);
    *L = F ? c.take<float>((size_t)du * du) : nullptr;
    *Linv = F ? c.take<float>((size_t)du * du) : nullptr;
    *Mb = F ? c.take<__nv_bfloat16>((size_t)du * pad8(du)) : nullptr;
    *work = F ? c.take<float>(cholesky_tc_work_bytes(du) / 4 + 1) : nullptr;
    *partial = c.take<float>(gram_partial_bytes(plan) / 4);
    *tiles = c.take<int2>(gram_tile_table_bytes(dv) / sizeof(int2) + 1);
    *lut = c.take<int>(gram_tile_table_bytes(dv) / sizeof(int) + 1);
    *Ptmp = accumulate ? c.take<float>((size_t)dv * dv) : nullptr;
  };
  DevStatus* st;
  __nv_bfloat16 *Ub, *Vb, *Mb;
  float *w, *L, *Linv, *work, *partial, *Ptmp;
  int2* tiles;
  int* lut;
  const size_t qpart_floats = qform_scratch_floats(N, du);
  {
    Carve c(nullptr);
    layout(c, &st, &Ub, &Vb, &w, &L, &Linv, &Mb, &work, &partial, &tiles, &lut, &Ptmp);
    c.take<float>(qpart_floats);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  layout(c, &st, &Ub, &Vb, &w, &L, &Linv, &Mb, &work, &partial, &tiles, &lut, &Ptmp);
  float* qpart = c.take<float>(qpart_floats);
  cudaStream_t s = h->stream;
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  CK(cudaMemsetAsync(w, 0, sizeof(float) * Npad, s));
  Staged us, vs_;
  ffh_status es = stage_input(h, U, true, N, du, Ub, nullptr, &us);
  if (es) return es;
  es = stage_input(h, V, true, N, dv, Vb, nullptr, &vs_);
  if (es) return es;
  // weights w_k = u_k^T F^-1 u_k (F = I: ||u_k||^2)
  if (F) {
    es = chol(h, F, du, L, Linv, work, st, 0);
    if (es) return es;
    es = qform(h, us, N, du, Linv, Mb, w, qpart, st);
    if (es) return es;
  } else {
    CK(launch_rowsumsq(us.raw, dtype, N, du, us.ld_raw, w, s));
  }
  GramTables gt;
  es = setup_tables(h, N, dv, &gt, tiles, lut);
  if (es) return es;
  es = gram(h, vs_, N, dv, w, 1.0f, accumulate ? Ptmp : P_out, partial, gt, st);
  if (es) return es;
  if (accumulate) CK(launch_add(P_out, Ptmp, dv * dv, s));
  DevStatus hst;
  es = read_status(h, st, &hst);
  if (logdet_F) *logdet_F = F ? hst.logdet : 0.0;
  return es;
}

extern "C" ffh_status ffh_update_from_sum(ffh_t h, const float* P, int64_t d, double scale,
                                          float* F_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  ffh_status vs = validate_opt(h);
  if (vs) return vs;
  if (!P || !F_out || d < 1 || !(scale > 0.0) || !std::isfinite(scale))
    return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (!is_device_ptr(P) || !is_device_ptr(F_out))
    return fail(h, FFH_ERR_INVALID_ARG, "ffh_update_from_sum takes device pointers");
  DevStatus* st;
  {
    Carve c(nullptr);
    c.take<DevStatus>(1);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  st = c.take<DevStatus>(1);
  cudaStream_t s = h->stream;
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  CK(launch_scale_copy(P, F_out, d * d, scale, s));
  CK(launch_damp(F_out, d, d, h->opt.damping, st, s));
  return read_status(h, st);
}

extern "C" ffh_status ffh_normalize_pair(ffh_t h, float* A, int64_t n, float* B, int64_t m,
                                         double* s_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  if (!A || !B || n < 1 || m < 1) return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (!is_device_ptr(A) || !is_device_ptr(B))
    return fail(h, FFH_ERR_INVALID_ARG, "ffh_normalize_pair takes device pointers");
  DevStatus* st;
  IterRecord* rec;
  {
    Carve c(nullptr);
    c.take<DevStatus>(1);
    c.take<IterRecord>(1);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  st = c.take<DevStatus>(1);
  rec = c.take<IterRecord>(1);
  cudaStream_t s = h->stream;
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  CK(launch_normalize(A, n, B, m, rec, st, s));
  IterRecord hr;
  CK(cudaMemcpyAsync(&hr, rec, sizeof(hr), cudaMemcpyDeviceToHost, s));
  ffh_status es = read_status(h, st);
  if (s_out) *s_out = hr.scale;
  return es;
}

extern "C" ffh_status ffh_relative_change(ffh_t h, const float* F, const float* Fprev, int64_t d,
                                          double* delta_out) {
  if (!h) return FFH_ERR_INVALID_ARG;
  h->err.clear();
  if (!F || !Fprev || !delta_out || d < 1) return fail(h, FFH_ERR_INVALID_ARG, "bad arguments");
  if (!is_device_ptr(F) || !is_device_ptr(Fprev))
    return fail(h, FFH_ERR_INVALID_ARG, "ffh_relative_change takes device pointers");
  DevStatus* st;
  double* acc;
  {
    Carve c(nullptr);
    c.take<DevStatus>(1);
    c.take<double>(4 + kRedDoubles);
    ffh_status es = ensure_ws(h, c.off + 1024);
    if (es) return es;
  }
  Carve c(h->ws);
  st = c.take<DevStatus>(1);
  acc = c.take<double>(4 + kRedDoubles);  // tr F, tr Fprev, d2, n2, then the scratch
  cudaStream_t s = h->stream;
  CK(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
  CK(launch_trace(F, d, acc + 0, s));
  CK(launch_trace(Fprev, d, acc + 1, s));
  CK(launch_delta(F, Fprev, d, acc + 2, acc + 3, acc, acc + 4, s));
  double hacc[4];
  CK(cudaMemcpyAsync(hacc, acc, sizeof(hacc), cudaMemcpyDeviceToHost, s));
  ffh_status es = read_status(h, st);
  *delta_out = hacc[3] > 0 ? std::sqrt(hacc[2] / hacc[3]) : 0.0;
  return es;
}
