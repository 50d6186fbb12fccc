// ffh_weighted_gram_static: the weighted Gram C = scale * V^T diag(w) V without any
// device allocation.
//
// Some callers cannot call cudaMalloc: code that runs inside a framework which owns
// every byte of device memory (a pre-reserved pool, an inference-engine plugin), or
// a latency-critical path where an allocation would synchronise the device.  This
// entry point therefore takes its working memory (the split-K partial tiles, the
// padded weights, the tile tables and the status word) from one file-scope device
// array of fixed size, and allocates nothing.  Only inputs and outputs come from the
// caller.
//
// The array lives as long as the library is loaded, on every GPU that loads it
// (kStaticScratchBytes each).  All calls share it and it keeps the contents of the
// last call: this file clears what must start at zero (status word, the weight tail
// beyond N) on every call.  Two calls whose work overlaps on the GPU (different
// streams, or different host threads) race on the array; callers must serialise them.
//
// Set-up: the first call on a device looks the array's device address up with
// cudaGetSymbolAddress (with that device current) and caches it; that first call
// should come before any stream capture.
#include <cstdio>
#include <mutex>

#include "ffh_internal.cuh"

namespace ffh {

static constexpr size_t kStaticScratchBytes = 64ull << 20;  // 64 MiB
static constexpr int kMaxDevices = 64;

// The scratch.  In host code this name is only a host-side stand-in for the symbol;
// kernels must be given the address returned by cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_gram_scratch[kStaticScratchBytes];

namespace {

std::mutex g_setup_mutex;
void* g_scratch_addr[kMaxDevices] = {};

void set_msg(char* buf, int32_t len, const char* msg) {
  if (!buf || len <= 0) return;
  int i = 0;
  for (; i < len - 1 && msg[i]; ++i) buf[i] = msg[i];
  buf[i] = 0;
}

__global__ void k_static_tiles(int64_t d, int nbm, int nbn, int2* tiles, int* lut) {
  // one thread: the tables are at most a few thousand entries
  if (blockIdx.x != 0 || threadIdx.x != 0) return;
  gram_fill_tiles(nbm, nbn, tiles, lut);
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

bool on_device(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

}  // namespace
}  // namespace ffh

using namespace ffh;

extern "C" ffh_status ffh_weighted_gram_static(const void* V, const float* w, int64_t N,
                                               int64_t d, float scale, float* C_out,
                                               void* cuda_stream, char* errbuf,
                                               int32_t errbuf_len) {
  if (!V || !C_out || N < 1 || d < 1 || d % 8 || N > ((int64_t)1 << 30)) {
    set_msg(errbuf, errbuf_len,
            "invalid arguments: need V, C_out, 1 <= N <= 2^30, d >= 1 a multiple of 8");
    return FFH_ERR_INVALID_ARG;
  }
  if (!on_device(V) || !on_device(C_out) || (w && !on_device(w))) {
    set_msg(errbuf, errbuf_len, "V, w and C_out must be device pointers");
    return FFH_ERR_INVALID_ARG;
  }
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    cudaGetLastError();
    set_msg(errbuf, errbuf_len, "no usable current CUDA device");
    return FFH_ERR_CUDA;
  }
  int major = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  if (major != 10) {
    set_msg(errbuf, errbuf_len, "needs a compute capability 10.x GPU");
    return FFH_ERR_UNSUPPORTED;
  }
  // the working-memory layout for this call; reject what does not fit
  const int64_t nbm = (d + kGramBM - 1) / kGramBM, nbn = (d + kGramBN - 1) / kGramBN;
  const int64_t Npad = (N + 63) / 64 * 64 + 64;
  GramPlan plan = gram_plan(N, d, num_sms());
  const size_t fixed = align256(sizeof(DevStatus)) + align256(sizeof(int2) * nbm * nbn) +
                       align256(sizeof(int) * nbm * nbn) + align256(sizeof(float) * Npad);
  while (plan.S > 1 && fixed + gram_partial_bytes(plan) > kStaticScratchBytes) {
    plan.S -= 1;
    plan.units = plan.T * plan.S;
    plan.grid = plan.units < num_sms() ? plan.units : num_sms();
  }
  if (fixed + gram_partial_bytes(plan) > kStaticScratchBytes) {
    char msg[256];
    snprintf(msg, sizeof(msg),
             "N=%lld, d=%lld needs %zu bytes of working memory; the static scratch holds %zu "
             "(d up to about 5000 fits)",
             (long long)N, (long long)d, fixed + gram_partial_bytes(plan), kStaticScratchBytes);
    set_msg(errbuf, errbuf_len, msg);
    return FFH_ERR_INVALID_ARG;
  }
  // set-up, once per device, with that device current
  unsigned char* base = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_addr[dev]) {
      void* p = nullptr;
      cudaError_t e = cudaGetSymbolAddress(&p, g_gram_scratch);
      if (e != cudaSuccess || !p) {
        cudaGetLastError();
        set_msg(errbuf, errbuf_len, "cudaGetSymbolAddress of the static scratch failed");
        return FFH_ERR_CUDA;
      }
      g_scratch_addr[dev] = p;
    }
    base = static_cast<unsigned char*>(g_scratch_addr[dev]);
  }
  size_t off = 0;
  DevStatus* st = reinterpret_cast<DevStatus*>(base + off);
  off += align256(sizeof(DevStatus));
  int2* tiles = reinterpret_cast<int2*>(base + off);
  off += align256(sizeof(int2) * nbm * nbn);
  int* lut = reinterpret_cast<int*>(base + off);
  off += align256(sizeof(int) * nbm * nbn);
  float* wpad = reinterpret_cast<float*>(base + off);
  off += align256(sizeof(float) * Npad);
  float* partial = reinterpret_cast<float*>(base + off);

  cudaError_t e = cudaMemsetAsync(st, 0, sizeof(DevStatus), s);
  const float* wuse = nullptr;
  if (e == cudaSuccess && w) {
    // the tail beyond N must read as zero (the array keeps the previous call's data)
    e = cudaMemcpyAsync(wpad, w, sizeof(float) * N, cudaMemcpyDeviceToDevice, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(wpad + N, 0, sizeof(float) * (Npad - N), s);
    wuse = wpad;
  }
  if (e == cudaSuccess) {
    k_static_tiles<<<1, 1, 0, s>>>(d, (int)nbm, (int)nbn, tiles, lut);
    note_launches(1);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess)
    e = launch_gram_tc(static_cast<const __nv_bfloat16*>(V), N, d, d, wuse, scale, C_out, d,
                       partial, tiles, lut, plan, st, 0, s);
  DevStatus hst;
  if (e == cudaSuccess) e = cudaMemcpyAsync(&hst, st, sizeof(hst), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) {
    set_msg(errbuf, errbuf_len, cudaGetErrorString(e));
    return FFH_ERR_CUDA;
  }
  if (hst.error) {
    set_msg(errbuf, errbuf_len, hst.error == FFH_ERR_TIMEOUT
                                    ? "a bounded device wait expired"
                                    : "device error");
    return static_cast<ffh_status>(hst.error);
  }
  set_msg(errbuf, errbuf_len, "");
  return FFH_OK;
}
