// k_fused.cu - the Gram pass (Eq. 9), the factor of A (Alg. 1 step 3) and the
// scores (Eq. 10) as roles of one persistent launch, so that each unit's
// values are read the second time (by the score role) soon after the first
// (by the Gram role), while L2 still holds them, instead of in a separate pass
// over the whole cache.
//
// One CTA per SM, all co-resident (a cooperative launch); CTA b takes a role:
//   b <  nf              factor role: units b, b + nf, ... (k_factor_body.cuh)
//   nf <= b < nf + ng    Gram role: items b - nf, b - nf + ng, ... (k_gram_body.cuh)
//   nf + ng <= b         score role: items b - nf - ng, ... + ns (k_score_body.cuh)
// Items are numbered unit-major, so each role sweeps the units in order and a
// unit's items are in flight at the same time. The roles meet through two
// per-unit counters of the workspace (zeroed by the plan kernel):
//   gcount[u]  every Gram item adds 6 once its data is visible device-wide
//              (each of the two weight warps for its weights, each of the
//              four epilogue warps for its rows of the partial Gram);
//   fdone[u]   set to 1 by the factor role once G, L^{-1} and the score
//              image of u are visible device-wide (it first waits for
//              gcount[u] = 6 x the unit's chunk count).
// The score role reads a unit's image and weights only after fdone[u]. No
// role waits on a later item of its own sequence and the Gram role waits on
// nothing, so with every CTA resident the schedule always progresses; each
// wait is bounded all the same (ST_TIMEOUT after WAIT_LIMIT_NS) and gives up
// early once another CTA has recorded a failure in the status word.
//
// L2: the Gram role loads the first `keep_tiles` V tiles of each item with the
// evict_last policy and the rest, and the logits/kappa rows, evict_first; the
// score role and the factor's partial reads are evict_first. The host sizes
// keep_tiles so that the evict_last lines in flight stay well inside L2.
#include "jacap_dev.cuh"
#include "jacap_internal.h"
#include "k_factor_body.cuh"
#include "k_gram_body.cuh"
#include "k_score_body.cuh"

namespace jacap {

constexpr int FU_THREADS = GR_THREADS;

template <int G>
constexpr size_t fused_smem_bytes() {
  constexpr size_t a = GrCfg<G, 1024>::SMEM, b = score_bf16_smem_bytes<false>(), c = FB_FUSED_SMEM;
  static_assert(FB_SMEM <= FB_FUSED_SMEM, "the factor's blocks fit in its staging ring");
  return a > b ? (a > c ? a : c) : (b > c ? b : c);
}

template <int G>
__global__ void __launch_bounds__(FU_THREADS, 1)
    fused_gfs_kernel(const __grid_constant__ CUtensorMap vmap, Dims dm, Ws ws, float* __restrict__ scores, int nf,
                     int ng) {
  pdl_wait();
  const int b = blockIdx.x;
  if (b < nf) {
    if (threadIdx.x < FB_THREADS) factor_blocked_cta<true>(dm, ws, b, nf);
  } else if (b < nf + ng) {
    gram_bf16_body<G, true>(&vmap, dm, ws, b - nf, ng);
  } else {
    score_bf16_body<false, true>(&vmap, dm, ws, scores, b - nf - ng, (int)gridDim.x - nf - ng);
  }
}

template <int G>
static cudaError_t launch_fused_g(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, float* scores,
                                  const FusedRoles& r, cudaStream_t st) {
  constexpr size_t smem = fused_smem_bytes<G>();
  static_assert(smem + 256 <= 232448, "shared memory of the fused kernel (256 B for static variables)");
  cudaError_t e = cudaFuncSetAttribute(fused_gfs_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(r.nf + r.ng + r.ns);
  cfg.blockDim = dim3(FU_THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // every CTA resident: the roles wait on one another
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  JACAP_TRY(cudaLaunchKernelEx(&cfg, fused_gfs_kernel<G>, vmap, dm, ws, scores, r.nf, r.ng));
  return cudaGetLastError();
}

cudaError_t launch_fused(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, float* scores, const FusedRoles& r,
                         cudaStream_t st) {
  if (r.nf < 1 || r.ng < 1 || r.ns < 1) return cudaErrorInvalidValue;
  switch (dm.G) {
    case 1: return launch_fused_g<1>(vmap, dm, ws, scores, r, st);
    case 2: return launch_fused_g<2>(vmap, dm, ws, scores, r, st);
    case 3: return launch_fused_g<3>(vmap, dm, ws, scores, r, st);
    case 4: return launch_fused_g<4>(vmap, dm, ws, scores, r, st);
    case 5: return launch_fused_g<5>(vmap, dm, ws, scores, r, st);
    case 6: return launch_fused_g<6>(vmap, dm, ws, scores, r, st);
    case 7: return launch_fused_g<7>(vmap, dm, ws, scores, r, st);
    case 8: return launch_fused_g<8>(vmap, dm, ws, scores, r, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace jacap
