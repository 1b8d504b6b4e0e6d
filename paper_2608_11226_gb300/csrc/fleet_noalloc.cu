// Fleet window accounting for callers that may not allocate device memory.
//
// Some callers cannot call cudaMalloc: code that runs inside a host process
// whose device memory belongs to another allocator (a training framework's
// caching allocator, a scheduler service holding a fixed memory budget), and
// control loops that must not add allocations, and the device-wide
// synchronisation an allocation may cause, to their own timeline.  This
// entry point runs the same kernels as pe_fleet_windows, but takes its
// scratch space from one file-scope device array of fixed size instead of a
// caller-provided workspace.
//
// The array lives in this translation unit's module.  Under lazy module
// loading (the CUDA default) the driver loads the module, and reserves the
// array on the current device, when the first call on that device looks up
// the array's address; from then on the device holds
// PE_FLEET_NOALLOC_SCRATCH_BYTES of it until the process exits.  That
// one-time reservation is the driver's; the calls themselves allocate
// nothing.  All calls share the array and it keeps the last call's contents;
// the kernels rewrite every word they read (the per-job sums) and the call
// clears the maxima and the error flag before use.  Calls that overlap on
// the GPU (on different streams, or from different host threads) race on
// the array.  Like pe_fleet_windows, every call waits on its stream for the
// device-side validation of the traces before it launches the counts.
#include <cuda.h>

#include <mutex>

#include "common.cuh"

namespace pe {

int64_t fleet_ws_min_bytes(int J, int L, int H);

static __device__ __align__(256) unsigned char g_fleet_scratch[PE_FLEET_NOALLOC_SCRATCH_BYTES];

// Device address of g_fleet_scratch per device ordinal, looked up once per
// device with that device current.  In host code the array's name is only a
// host-side stand-in, never a device address.  The address belongs to the
// context that loaded the module: the cache records that context's unique
// id and looks the address up again when the device's current context is a
// different one (after cudaDeviceReset, or a primary-context reset).
typedef CUresult(CUDAAPI* CtxGetCurrentFn)(CUcontext*);
typedef CUresult(CUDAAPI* CtxGetIdFn)(CUcontext, unsigned long long*);

struct ScratchSlot {
  void* ptr = nullptr;
  unsigned long long ctx_id = 0;
};

static std::mutex g_scratch_mu;
static ScratchSlot g_scratch[256];
static CtxGetCurrentFn g_ctx_current = nullptr;
static CtxGetIdFn g_ctx_id = nullptr;

static pe_status current_context_id(unsigned long long* id) {
  if (!g_ctx_current || !g_ctx_id) {
    void* f0 = nullptr;
    void* f1 = nullptr;
    cudaDriverEntryPointQueryResult q0, q1;
    PE_TRY_CUDA(cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f0, 12000, cudaEnableDefault, &q0));
    PE_TRY_CUDA(cudaGetDriverEntryPointByVersion("cuCtxGetId", &f1, 12000, cudaEnableDefault, &q1));
    if (q0 != cudaDriverEntryPointSuccess || q1 != cudaDriverEntryPointSuccess || !f0 || !f1)
      return fail(PE_ECUDA, "the CUDA driver does not provide cuCtxGetCurrent / cuCtxGetId");
    g_ctx_current = reinterpret_cast<CtxGetCurrentFn>(f0);
    g_ctx_id = reinterpret_cast<CtxGetIdFn>(f1);
  }
  CUcontext ctx = nullptr;
  if (g_ctx_current(&ctx) != CUDA_SUCCESS || !ctx) return fail(PE_ECUDA, "no current CUDA context");
  if (g_ctx_id(ctx, id) != CUDA_SUCCESS) return fail(PE_ECUDA, "cuCtxGetId failed");
  return PE_OK;
}

static pe_status scratch_address(void** out) {
  int dev = 0;
  PE_TRY_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 256) return fail(PE_EINVAL, "device ordinal %d out of range", dev);
  // cudaSetDevice makes the device's primary context current (initialising
  // it on first use), so the context id below is the one the runtime
  // launches into
  PE_TRY_CUDA(cudaSetDevice(dev));
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  unsigned long long id = 0;
  pe_status s = current_context_id(&id);
  if (s != PE_OK) return s;
  ScratchSlot& slot = g_scratch[dev];
  if (!slot.ptr || slot.ctx_id != id) {
    void* p = nullptr;
    PE_TRY_CUDA(cudaGetSymbolAddress(&p, g_fleet_scratch));
    slot.ptr = p;
    slot.ctx_id = id;
  }
  *out = slot.ptr;
  return PE_OK;
}

}  // namespace pe

extern "C" pe_status pe_fleet_windows_noalloc(const float* traces, int32_t G, int32_t L,
                                              const int32_t* job_of_gpu, int32_t J,
                                              const int32_t* offsets, int64_t N, int32_t H,
                                              const int32_t* windows, int32_t W,
                                              int64_t budget_q, int32_t* counts, int32_t* peaks,
                                              void* stream) {
  using namespace pe;
  clear_error();
  if (J < 1 || J > 32 || L < 1 || H < 0) return fail(PE_EINVAL, "J must be in [1, 32], L >= 1, H >= 0");
  const int64_t need = fleet_ws_min_bytes(J, L, H);
  if (need > (int64_t)PE_FLEET_NOALLOC_SCRATCH_BYTES)
    return fail(PE_EINVAL,
                "fleet scratch of %lld bytes (one prefix copy) exceeds the fixed %lld-byte "
                "static scratch of pe_fleet_windows_noalloc; use pe_fleet_windows with a workspace",
                (long long)need, (long long)PE_FLEET_NOALLOC_SCRATCH_BYTES);
  void* scratch = nullptr;
  pe_status s = scratch_address(&scratch);
  if (s != PE_OK) return s;
  return pe_fleet_windows(traces, G, L, job_of_gpu, J, offsets, N, H, windows, W, budget_q, counts,
                          peaks, scratch, (int64_t)PE_FLEET_NOALLOC_SCRATCH_BYTES, stream);
}
