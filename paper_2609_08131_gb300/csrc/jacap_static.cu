// jacap_static.cu - jacap_score_static: the scoring pass with its workspace in
// library-owned static device memory (declared in include/jacap.h).
//
// Some callers cannot allocate device memory at the point where they score: a
// serving loop that owns a fixed arena, or code that must not grow the memory
// footprint after start-up. For them the library keeps one fixed scratch array
// per device, sized at link time, and runs the ordinary scoring kernels on it.
// The paper describes no such entry point; it is a deployment convenience.
//
// Nothing here allocates: the scratch is a file-scope __device__ array that
// the CUDA runtime places with the module. Set-up happens once per device (and
// again whenever that device's current context is a different one, e.g. after
// cudaDeviceReset): with the device current, cudaGetSymbolAddress gives the
// array's device address in that context, which is cached together with the
// context's id. The work is then exactly that of jacap_score on that address.
#include <cudaTypedefs.h>
#include <mutex>

#include "jacap.h"

namespace {

// The scratch, one copy per device context (the module is loaded per context).
static __device__ __align__(256) unsigned char g_static_scratch[JACAP_STATIC_SCRATCH_BYTES];

constexpr int MAX_DEVICES = 64;
struct Slot {
  unsigned long long ctx_id;  // id of the context the address belongs to (0: none yet)
  void* addr;
};
std::mutex g_setup_mutex;
Slot g_slot[MAX_DEVICES] = {};

// Id of the calling thread's current context, or 0 if there is none (the
// runtime has not made one current yet) or the driver calls are unavailable.
unsigned long long current_context_id() {
  static PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
  static PFN_cuCtxGetId_v12000 get_id = nullptr;
  static bool resolved = false;
  if (!resolved) {  // called under g_setup_mutex
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = (PFN_cuCtxGetCurrent_v4000)p;
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = (PFN_cuCtxGetId_v12000)p;
    resolved = true;
  }
  if (get_current == nullptr || get_id == nullptr) return 0;
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr || get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Address of the scratch in the current device's context, or NULL if the
// lookup fails. Looked up on the first call per device (that device current)
// and whenever the current context is not the one the cached address belongs
// to; the first lookup in a context loads the module's static memory.
void* scratch_for_current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= MAX_DEVICES) return nullptr;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  Slot& slot = g_slot[dev];
  const unsigned long long id = current_context_id();
  if (slot.addr != nullptr && id != 0 && slot.ctx_id == id) return slot.addr;
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr) return nullptr;
  // the lookup made the device's context current if it was not yet
  slot.ctx_id = current_context_id();
  slot.addr = slot.ctx_id != 0 ? p : nullptr;  // without a context id, look up again next time
  return p;
}

}  // namespace

extern "C" {

jacap_status jacap_score_static(const jacap_layout* layout, const jacap_params* params, const void* q_win,
                                const void* k, const void* v, float* scores, void* stream, void** scratch_out) {
  // Size first, so an oversized layout is refused before any CUDA call.
  const size_t need = jacap_workspace_size(layout, 1);
  // An invalid or unsupported layout: jacap_score reports which, from its
  // host checks, before it looks at the (absent) workspace.
  if (need == 0) return jacap_score(layout, params, q_win, k, v, scores, nullptr, 0, stream);
  if (need > (size_t)JACAP_STATIC_SCRATCH_BYTES) return JACAP_ERR_WORKSPACE;
  void* ws = scratch_for_current_device();
  if (ws == nullptr) return JACAP_ERR_CUDA;
  if (scratch_out != nullptr) *scratch_out = ws;
  // jacap_score's first kernel clears the status word (the only state that
  // must start at zero); every other section of the workspace is written
  // before it is read within one pass.
  return jacap_score(layout, params, q_win, k, v, scores, ws, (size_t)JACAP_STATIC_SCRATCH_BYTES, stream);
}

}  // extern "C"
