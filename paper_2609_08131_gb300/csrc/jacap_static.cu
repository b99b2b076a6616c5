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
// the CUDA runtime places with the module, its address is looked up once per
// device with cudaGetSymbolAddress, and the work is then exactly that of
// jacap_score on that address.
#include <mutex>

#include "jacap.h"

namespace {

// The scratch, one copy per device context (the module is loaded per device).
static __device__ __align__(256) unsigned char g_static_scratch[JACAP_STATIC_SCRATCH_BYTES];

constexpr int MAX_DEVICES = 64;
std::mutex g_setup_mutex;
void* g_scratch_addr[MAX_DEVICES] = {};

// Address of this device's scratch; looked up on the first call per device
// (with that device current) and cached. Returns NULL on failure.
void* scratch_for_current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= MAX_DEVICES) return nullptr;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr) return nullptr;
    g_scratch_addr[dev] = p;
  }
  return g_scratch_addr[dev];
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
