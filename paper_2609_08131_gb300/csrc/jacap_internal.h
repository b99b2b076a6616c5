// jacap_internal.h - host-side launchers of the libjacap kernels.
// All launchers enqueue on `st` and return the launch error (cudaSuccess if
// the kernel was enqueued).
#pragma once

#include "jacap_dev.cuh"

namespace jacap {

// Tracing: built with -DJACAP_NVTX (JACAP_NVTX=1 in the environment of the
// build), the host side marks each kernel's launch with an NVTX range named
// "jacap/<step>" so a profiler timeline groups the GPU work by step of the
// pass; otherwise the ranges compile to nothing.
#ifdef JACAP_NVTX
#include <nvtx3/nvToolsExt.h>
inline void trace_push(const char* name) { nvtxRangePushA(name); }
inline void trace_pop() { nvtxRangePop(); }
#else
inline void trace_push(const char*) {}
inline void trace_pop() {}
#endif
struct TraceRange {
  explicit TraceRange(const char* name) { trace_push(name); }
  ~TraceRange() { trace_pop(); }
  TraceRange(const TraceRange&) = delete;
  TraceRange& operator=(const TraceRange&) = delete;
};

// Returns a failed CUDA call's error from the enclosing launcher.
#define JACAP_TRY(call)                     \
  do {                                      \
    const cudaError_t e_ = (call);          \
    if (e_ != cudaSuccess) return e_;       \
  } while (0)

// Launch `kernel`, with programmatic stream serialization when `pdl` (see
// pdl_wait()): the launch is prepared while the previous kernel of the stream
// runs and the kernel waits for it inside. Returns the launch error.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(bool pdl, void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = pdl ? attr : nullptr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

cudaError_t launch_plan(const Dims& dm, const Ws& ws, const int32_t* cu, cudaStream_t st);
cudaError_t launch_window_stats(const Dims& dm, const Ws& ws, int dtype, const void* q, cudaStream_t st);
cudaError_t launch_kpass(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int dtype, const int32_t* cu,
                         int grid, cudaStream_t st);
cudaError_t launch_kpass_bf16(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, const int32_t* cu, int grid,
                              cudaStream_t st);
// Full covariance (App. B.2): with a bf16 cache and a supported window shape
// (kfull_uses_tensor_cores) launch_kpass_full replaces the K pass (logits,
// full-covariance kappa and softmax statistics in one read of K); otherwise
// the K pass runs and launch_kfull (CUDA cores) overwrites its diagonal kappa.
bool kfull_uses_tensor_cores(const Dims& dm, int dtype);
cudaError_t launch_kpass_full(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int grid, cudaStream_t st);
// one thread waits (bounded by limit_ns) on an mbarrier nothing arrives on
cudaError_t launch_selftest_wait(const Ws& ws, unsigned long long limit_ns, cudaStream_t st);
cudaError_t launch_kfull(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int dtype, const void* k, int grid,
                         cudaStream_t st);
// The pool-softmax normaliser (M_h, 1 / Z_h) of every unit and query head,
// merged once from the K pass's chunk statistics into ws.ustats.
cudaError_t launch_unit_stats(const Dims& dm, const Ws& ws, cudaStream_t st);
cudaError_t launch_weights(const Dims& dm, const Ws& ws, const int32_t* cu, int grid, cudaStream_t st);
cudaError_t launch_gram(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, int dtype, const void* v,
                        const int32_t* cu, int grid, cudaStream_t st);
cudaError_t launch_factor(const Dims& dm, const Ws& ws, const float* out_factor, cudaStream_t st);
cudaError_t launch_score(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, int dtype, const void* v,
                         const int32_t* cu, float* scores, int grid, cudaStream_t st);
// The fused schedule (k_fused.cu): CTAs of the factor, Gram and score roles.
struct FusedRoles {
  int nf, ng, ns;
};
// Gram, factor and scores of a bf16 cache in one cooperative launch of
// nf + ng + ns CTAs (at most one per SM); dm.keep_tiles set by the caller.
cudaError_t launch_fused(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, float* scores, const FusedRoles& r,
                         cudaStream_t st);
// Selection only when k and kio are null. With k: the kept rows of k and v
// (dtype 1 = bf16, 0 = float32) are also copied into k_out and v_out, as
// launch_compact does. With kio: the holes of kio, vio (and pos) are filled in
// place, as launch_compact_inplace does without preserve_order.
cudaError_t launch_select(const Dims& dm, const Ws& ws, const int32_t* cu, const float* scores, int budget,
                          int32_t* idx, int32_t* kept, int max_seqlen, int grid, cudaStream_t st, int dtype = 1,
                          const void* k = nullptr, const void* v = nullptr, void* k_out = nullptr,
                          void* v_out = nullptr, void* kio = nullptr, void* vio = nullptr, int32_t* pos = nullptr);
cudaError_t launch_compact(const Dims& dm, int dtype, const int32_t* cu, const void* k, const void* v,
                           const int32_t* idx, int budget, void* k_out, void* v_out, cudaStream_t st);
cudaError_t launch_stats_update(const Dims& dm, int dtype, const void* q, float* stats, int32_t* counts, int reset,
                                cudaStream_t st);
cudaError_t launch_stats_moments(const Dims& dm, const Ws& ws, const float* stats, const int32_t* counts,
                                 cudaStream_t st);
cudaError_t launch_compact_inplace(const Dims& dm, const Ws& ws, int dtype, const int32_t* cu, void* k, void* v,
                                   int32_t* pos, const int32_t* idx, int budget, int preserve_order,
                                   cudaStream_t st);

}  // namespace jacap
