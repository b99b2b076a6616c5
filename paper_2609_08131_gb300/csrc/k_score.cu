// k_score.cu - Jacap scores r_i = w_i v_i^T A^{-1} v_i = w_i ||L^{-1} v_i||^2 (Eq. 10).
//
// bf16 caches: the tensor cores form Y = V (L^{-1})^T for a 128-token tile
// from hi(L^{-1}) and lo(L^{-1}) (K-major, from a 64 KB shared-memory image
// written by the factor kernel, hi and lo interleaved by 16-row blocks).
// L^{-1} is lower triangular, so output row n needs only channels <= n: the
// K-step of channels 16 k .. 16 k + 15 is one MMA of N = 256 - 32 k over the
// image rows (hi and lo of output rows 16 k .. 127) into accumulator columns
// 32 k .. 255, eight MMAs per tile in all. The image's rows 0-127 of channels
// 64-127 (output rows 0-63) are zero and not copied into shared memory, which
// leaves room for a fourth V stage. V comes straight from the TMA-staged tile;
// a warp of its own loads the images, so the V ring never waits behind an
// image slot. Each epilogue thread owns one token (one TMEM lane) and reduces
// ||y||^2 = sum_n (hi_n + lo_n)^2 in fp32, then multiplies by w_i. (With
// output directions the matrix is full: hi and lo accumulate into the same
// 128 columns, four MMAs of N = 128 per K-step pair.) The tensor-memory accumulator
// is double-buffered so the epilogue of tile i overlaps the MMAs of tile i+1,
// and so is the L^{-1} image: it is loaded once per run of consecutive items
// of one unit, and the next unit's image streams in while the current run's
// tiles go through.
// float32 caches: SIMT forward products with L^{-1} held in shared memory.
#include "jacap_dev.cuh"
#include "jacap_internal.h"
#include "k_score_body.cuh"

namespace jacap {

template <bool DENSE>
__global__ void __launch_bounds__(SC_THREADS, 1)
    score_bf16_kernel(const __grid_constant__ CUtensorMap vmap, Dims dm, Ws ws, const int32_t* __restrict__ cu,
                      float* __restrict__ scores) {
  pdl_wait();
  score_bf16_body<DENSE, false>(&vmap, dm, ws, scores, blockIdx.x, gridDim.x);
}

// ------------------------------------------------------------ SIMT fp32 ---
// Two threads per token (lanes 2 t and 2 t + 1): thread `half` forms the
// output rows r of the quads r / 4 = half, half + 2, ... (the two halves of
// the triangle get about the same work), four rows at once so their
// multiply-add chains interleave, and the pair adds its squared norms.
// L^{-1} is stored with zeros above the diagonal, so a quad may run its
// columns up to its last row. Four columns per step: one 16-byte load of each
// of the quad's rows and of the token's row serves 16 multiply-adds (the
// staged rows are 16-byte aligned).
constexpr int SF_THREADS = 2 * TILE;
constexpr int SF_LD = D + 4;
constexpr size_t score_f32_smem_bytes() { return (size_t)(D * D + TILE * SF_LD) * sizeof(float); }

__global__ void __launch_bounds__(SF_THREADS)
    score_f32_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu, const float* __restrict__ v,
                     float* __restrict__ scores) {
  pdl_wait();
  extern __shared__ __align__(16) float ssm[];
  float* Mi = ssm;               // [D][D] L^{-1}
  float* vt = ssm + D * D;       // [TILE][SF_LD]
  __shared__ int s_skip;
  const int tid = threadIdx.x;
  if (tid == 0) s_skip = status_failed(ws) ? 1 : 0;
  __syncthreads();
  if (s_skip) return;
  const int tk = tid >> 1, half = tid & 1;
  bool bad = false;
  int64_t loaded = -1;
  Item item;
  for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
    const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
    const int64_t u = (int64_t)item.plane * dm.S + item.seq;
    const float* vbase = v + (int64_t)l * dm.kv_sl + (int64_t)g * dm.kv_sh;
    __syncthreads();
    if (u != loaded) {
      // unrolled so that all of a thread's loads are in flight before its stores
      const float* src = ws.minv + u * D * D;
#pragma unroll
      for (int e = tid * 4; e < D * D; e += SF_THREADS * 4) *(float4*)(Mi + e) = *(const float4*)(src + e);
      loaded = u;
    }
    for (int64_t t = item.t0; t < item.t1; t += TILE) {
      __syncthreads();
#pragma unroll
      for (int e = tid; e < TILE * (D / 4); e += SF_THREADS) {
        const int r = e / (D / 4), c4 = (e % (D / 4)) * 4;
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (t + r < item.t1) x = *(const float4*)(vbase + (t + r) * dm.kv_st + c4);
        *(float4*)(vt + r * SF_LD + c4) = x;
      }
      __syncthreads();
      const float* vr = vt + tk * SF_LD;
      float ssq = 0.f;
      for (int r0 = 4 * half; r0 < D; r0 += 8) {
        const float* m0 = Mi + r0 * D;
        // a full matrix with output directions
        const int cend = dm.dense_minv ? D : r0 + 4;
        float y0 = 0.f, y1 = 0.f, y2 = 0.f, y3 = 0.f;
        for (int c = 0; c < cend; c += 4) {  // cend is a multiple of 4
          const float4 x = *(const float4*)(vr + c);
          const float4 a0 = *(const float4*)(m0 + c), a1 = *(const float4*)(m0 + D + c);
          const float4 a2 = *(const float4*)(m0 + 2 * D + c), a3 = *(const float4*)(m0 + 3 * D + c);
          y0 = fmaf(a0.x, x.x, y0), y1 = fmaf(a1.x, x.x, y1), y2 = fmaf(a2.x, x.x, y2), y3 = fmaf(a3.x, x.x, y3);
          y0 = fmaf(a0.y, x.y, y0), y1 = fmaf(a1.y, x.y, y1), y2 = fmaf(a2.y, x.y, y2), y3 = fmaf(a3.y, x.y, y3);
          y0 = fmaf(a0.z, x.z, y0), y1 = fmaf(a1.z, x.z, y1), y2 = fmaf(a2.z, x.z, y2), y3 = fmaf(a3.z, x.z, y3);
          y0 = fmaf(a0.w, x.w, y0), y1 = fmaf(a1.w, x.w, y1), y2 = fmaf(a2.w, x.w, y2), y3 = fmaf(a3.w, x.w, y3);
        }
        ssq = fmaf(y0, y0, fmaf(y1, y1, fmaf(y2, y2, fmaf(y3, y3, ssq))));
      }
      ssq += __shfl_xor_sync(0xffffffffu, ssq, 1);
      const int64_t tok = t + tk;
      if (half == 0 && tok < item.t1) {
        const int64_t o = (int64_t)item.plane * dm.Ntot + tok;
        const float sc = ws.w[o] * ssq;
        scores[o] = sc;
        bad |= !isfinite(sc);
      }
    }
  }
  if (bad) flag(ws, ST_NONFINITE);
}

cudaError_t launch_score(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, int dtype, const void* v,
                         const int32_t* cu, float* scores, int grid, cudaStream_t st) {
  if (dtype == 1) {
    const size_t smem = dm.dense_minv ? score_bf16_smem_bytes<true>() : score_bf16_smem_bytes<false>();
    static_assert(score_bf16_smem_bytes<true>() <= 232448 && score_bf16_smem_bytes<false>() <= 232448, "smem");
    auto kern = dm.dense_minv ? score_bf16_kernel<true> : score_bf16_kernel<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    JACAP_TRY(launch_pdl(dm.pdl != 0, kern, grid, SC_THREADS, smem, st, vmap, dm, ws, cu, scores));
  } else {
    constexpr size_t smem = score_f32_smem_bytes();
    cudaError_t e = cudaFuncSetAttribute(score_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    JACAP_TRY(launch_pdl(dm.pdl != 0, score_f32_kernel, grid, SF_THREADS, smem, st, dm, ws, cu, (const float*)v,
                         scores));
  }
  return cudaGetLastError();
}

}  // namespace jacap
