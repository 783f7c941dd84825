// bag_rel_l1_noalloc: the trajectory-signal reduction of bag_rel_l1 without any
// allocation, for callers that cannot call cudaMalloc.
//
// Who cannot allocate: code embedded in a host framework whose caching allocator has
// already reserved the device's memory and does not allow raw cudaMalloc calls next to
// it, and latency-critical loops that cannot afford the implicit device-wide
// synchronisation that cudaMalloc / cudaFree may perform.  They also cannot create a
// bag context (bag_create allocates), so this entry point takes no context: the caller
// passes the inputs, the output and a stream.
//
// The per-row partial sums that bag_rel_l1 keeps in caller-provided scratch live here
// in a fixed-size file-scope device array instead.  Every GPU that loads the library
// holds that array (2 * kNoAllocMaxRows floats = 512 KiB) until the process exits.
// In host code the array's name stands for a host-side shadow, not a device address, so
// the device address is looked up with cudaGetSymbolAddress once per device, on the
// first call made while that device is current; make that first call before any stream
// capture.  The cached address belongs to the CUDA context it was looked up in: it is
// kept with that context's unique id and looked up again when the device's current
// context changes (after cudaDeviceReset, or when the primary context is re-created).  Every call shares the array and it keeps the last call's contents; each call
// writes every entry it later reads, so nothing has to start at zero.  Calls whose
// kernels overlap on the GPU (e.g. on two unordered streams) race on the array.
#include <mutex>
#include <string>

#include "bag.h"
#include "kernels.h"

namespace {
constexpr long kNoAllocMaxRows = 65536;
constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
// per device: the scratch address and the id of the context it was looked up in
float* g_scratch_ptr[kMaxDevices] = {nullptr};
unsigned long long g_scratch_ctx[kMaxDevices] = {0};

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

// Unique id of the calling thread's current CUDA context (0 when none is current or the
// driver does not provide the query).
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  if (!get_current || !get_id) return 0;
  CUcontext c = nullptr;
  unsigned long long id = 0;
  if (get_current(&c) != CUDA_SUCCESS || !c || get_id(c, &id) != CUDA_SUCCESS) return 0;
  return id;
}
}  // namespace

static __device__ __align__(256) float g_rel_l1_scratch[2 * kNoAllocMaxRows];

// Device address of the scratch array in the current device's current context (looked
// up once per context).
static bag_status noalloc_scratch(float** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    bag::set_global_error("bag_rel_l1_noalloc: cudaGetDevice failed");
    return BAG_ECUDA;
  }
  if (dev < 0 || dev >= kMaxDevices) {
    bag::set_global_error("bag_rel_l1_noalloc: device ordinal out of range");
    return BAG_EUNSUPPORTED;
  }
  std::lock_guard<std::mutex> lock(g_setup_mu);
  const unsigned long long id = current_context_id();
  if (!g_scratch_ptr[dev] || id == 0 || id != g_scratch_ctx[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_rel_l1_scratch);
    if (e != cudaSuccess || !p) {
      g_scratch_ptr[dev] = nullptr;
      bag::set_global_error(std::string("bag_rel_l1_noalloc: cudaGetSymbolAddress failed: ") +
                            cudaGetErrorString(e));
      return BAG_ECUDA;
    }
    g_scratch_ptr[dev] = static_cast<float*>(p);
    // the look-up makes the device's primary context current if none was
    g_scratch_ctx[dev] = id ? id : current_context_id();
  }
  *out = g_scratch_ptr[dev];
  return BAG_OK;
}

extern "C" bag_status bag_rel_l1_noalloc(const void* a, const void* b, int dtype, long rows,
                                         long cols, float* out, void* cuda_stream) {
  if (!a || !b || !out) {
    bag::set_global_error("bag_rel_l1_noalloc: null pointer");
    return BAG_EINVAL;
  }
  if (rows <= 0 || cols <= 0 || (dtype != BAG_F32 && dtype != BAG_BF16)) {
    bag::set_global_error("bag_rel_l1_noalloc: bad shape or dtype");
    return BAG_EINVAL;
  }
  if (rows > kNoAllocMaxRows) {
    bag::set_global_error("bag_rel_l1_noalloc: rows = " + std::to_string(rows) +
                          " exceeds the fixed scratch limit of " +
                          std::to_string(kNoAllocMaxRows) + " rows");
    return BAG_EINVAL;
  }
  float* scratch = nullptr;
  const bag_status s = noalloc_scratch(&scratch);
  if (s != BAG_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  cudaError_t e = bag::rel_l1_partials(a, b, dtype == BAG_BF16, rows, cols, scratch, st);
  if (e == cudaSuccess) e = bag::rel_l1_finalize(scratch, rows, out, st);
  if (e != cudaSuccess) {
    bag::set_global_error(std::string("bag_rel_l1_noalloc: ") + cudaGetErrorString(e));
    return BAG_ECUDA;
  }
  return BAG_OK;
}
