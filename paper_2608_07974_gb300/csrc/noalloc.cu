// Allocation-free variant of the fused local-objective entry point (zl_op_local_loss).
//
// Some callers cannot call cudaMalloc: a host framework whose caching allocator has reserved the
// whole device budget (an outside cudaMalloc then fails or breaks its accounting), or a
// latency-critical loop that must not take the device-wide synchronisation cudaMalloc/cudaFree
// can imply. This entry point keeps its scratch (per-row losses, |Omega|, an error word) in a
// file-scope __device__ array instead, so it allocates nothing; the caller still passes every
// input and output.
//
// The array is a host-side stand-in in host code, not a device address: the address handed to
// the kernels comes from cudaGetSymbolAddress, looked up with the device current by the first call
// in each CUDA context (the cache is keyed on the context's process-unique id, so a context created
// after cudaDeviceReset, or a caller's own context, gets its own lookup). Every call shares the
// array, so calls whose work overlaps on the GPU race on it; |Omega| and the error word are written
// before they are read on each call, the per-row losses are fully rewritten.
#include <cuda.h>
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "common.cuh"
#include "ops.h"
#include "zerolock.h"

namespace {

constexpr int kMaxRows = ZL_NOALLOC_MAX_ROWS;
constexpr int kCountSlot = kMaxRows;        // |Omega| (int), 256-byte aligned
constexpr int kErrSlot = kMaxRows + 64;     // device-side argument error bits
static __device__ __align__(256) float g_scratch[kMaxRows + 128];

std::mutex g_mu;
struct CtxAddr {
  unsigned long long ctx_id;
  void* addr;
};
constexpr int kMaxContexts = 64;
CtxAddr g_addr[kMaxContexts];
int g_naddr = 0;

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

template <typename F>
F driver_fn(const char* name) {
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess)
    return nullptr;
  return reinterpret_cast<F>(fn);
}

// Id of the calling thread's current CUDA context (0 if there is none or it cannot be read).
unsigned long long current_ctx_id() {
  static CtxGetCurrentFn get_cur = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent");
  static CtxGetIdFn get_id = driver_fn<CtxGetIdFn>("cuCtxGetId");
  CUcontext cx = nullptr;
  unsigned long long id = 0;
  if (!get_cur || !get_id || get_cur(&cx) != CUDA_SUCCESS || !cx || get_id(cx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

zl_status fail(zl_status st, const std::string& m) {
  zl::set_last_error(m);
  return st;
}

}  // namespace

extern "C" zl_status zl_op_local_loss_noalloc(int dtype, const void* z, const void* t, const int32_t* labels, int N,
                                              int V, int ldz, float alpha, int kl_dir, void* dz, float* loss,
                                              void* stream) {
  if (!z || !labels || !dz || !loss) return fail(ZL_ERR_ARG, "NULL argument");
  if (dtype != 0 && dtype != 1) return fail(ZL_ERR_ARG, "dtype must be ZL_DTYPE_F32 or ZL_DTYPE_BF16");
  if (N < 1 || V < 2 || ldz < V || ldz % 8 != 0) return fail(ZL_ERR_ARG, "need N >= 1, V >= 2, ldz >= V, ldz % 8 == 0");
  if (N > kMaxRows)
    return fail(ZL_ERR_ARG, "zl_op_local_loss_noalloc: N = " + std::to_string(N) + " exceeds the scratch limit of " +
                                std::to_string(kMaxRows) + " rows");
  if (!(alpha > 0.f && alpha <= 1.f) || (alpha < 1.f && !t) || (kl_dir != 0 && kl_dir != 1))
    return fail(ZL_ERR_ARG, "alpha in (0,1], t required when alpha < 1, kl_dir 0/1");
  float* base = nullptr;
  cudaError_t e = cudaSuccess;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    const unsigned long long id = current_ctx_id();
    for (int i = 0; id && i < g_naddr; ++i)
      if (g_addr[i].ctx_id == id) base = static_cast<float*>(g_addr[i].addr);
    if (!base) {   // first call in this context: look the array up with the device current
      void* p = nullptr;
      e = cudaGetSymbolAddress(&p, g_scratch);
      if (e != cudaSuccess || !p)
        return fail(ZL_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
      base = static_cast<float*>(p);
      const unsigned long long id2 = current_ctx_id();   // the lookup may have made the context current
      if (id2 && g_naddr < kMaxContexts) g_addr[g_naddr++] = CtxAddr{id2, p};
    }
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* row_loss = base;
  int* count = reinterpret_cast<int*>(base + kCountSlot);
  unsigned* err = reinterpret_cast<unsigned*>(base + kErrSlot);
  e = cudaMemsetAsync(err, 0, sizeof(unsigned), s);
  if (e != cudaSuccess) return fail(ZL_ERR_CUDA, std::string("cudaMemsetAsync: ") + cudaGetErrorString(e));
  zl::launch_count_valid(labels, N, V, count, err, s);
  zl::launch_local_loss(dtype, z, alpha < 1.f ? t : nullptr, labels, N, V, ldz, alpha, kl_dir, count, dz, row_loss, s);
  zl::launch_loss_reduce(row_loss, N, count, loss, s);
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(ZL_ERR_CUDA, std::string("launch: ") + cudaGetErrorString(e));
  return ZL_OK;
}
