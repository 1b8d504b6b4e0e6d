// Fleet window accounting for callers that may not allocate device memory.
//
// Some callers cannot call cudaMalloc: code that runs inside a host process
// whose device memory belongs to another allocator (a training framework's
// caching allocator, a scheduler service holding a fixed memory budget), and
// control loops that cannot afford the device-wide synchronisation an
// allocation may cause.  This entry point runs the same kernels as
// pe_fleet_windows, but takes its scratch space from one file-scope device
// array of fixed size instead of a caller-provided workspace.
//
// The array lives in the library's module: every GPU that loads the library
// holds PE_FLEET_NOALLOC_SCRATCH_BYTES of it until the process exits.  All
// calls share it and it keeps the last call's contents; the kernels rewrite
// every word they read (the per-job sums) and the call clears the maxima and
// the error flag before use.  Calls that overlap on the GPU (on different
// streams, or from different host threads) race on the array.
#include <mutex>

#include "common.cuh"

namespace pe {

int64_t fleet_ws_min_bytes(int J, int L, int H);

static __device__ __align__(256) unsigned char g_fleet_scratch[PE_FLEET_NOALLOC_SCRATCH_BYTES];

// device address of g_fleet_scratch per device ordinal; in host code the
// array's name is only a host-side stand-in, never a device address
static std::mutex g_scratch_mu;
static void* g_scratch_ptr[256] = {};

static pe_status scratch_address(void** out) {
  int dev = 0;
  PE_TRY_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 256) return fail(PE_EINVAL, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    PE_TRY_CUDA(cudaGetSymbolAddress(&p, g_fleet_scratch));
    g_scratch_ptr[dev] = p;
  }
  *out = g_scratch_ptr[dev];
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
