// k_gram.cu - Jacobian weights and the weighted Gram pass over V.
//
// Weight pass (one streaming pass over the K pass's logits/kappa rows), per
// work item (a chunk of one unit's tokens):
//   1. combines the K pass's per-chunk (max, sum exp) into the pool-softmax
//      normaliser (M_h, Z_h) of each query head h of the group (Sec. 3.4,
//      display after Algorithm 1);
//   2. forms w_i = (1/d) sum_h [alpha_bar (1 - alpha_bar)]^2 kappa_h,i with
//      alpha_bar = exp(l_h,i - M_h) / Z_h (Eq. 8; GQA heads summed) and stores
//      w for the score pass and as a bf16 pair hi + lo for the Gram pass.
// Gram pass: accumulates the chunk's partial Gram  sum_i w_i v_i v_i^T  (Eq. 9).
//
// bf16 caches use the 5th-generation tensor cores. B = V straight from the
// TMA-staged tile (bf16 is exact); the scaled operand w_i v_i = hi + lo is
// split into two bf16 halves (residual ~2^-17 relative per product) by the
// scaling warps with packed bf16 arithmetic on w_i = whi + wlo, and written to
// tensor memory as two A operands, so
// D = sum_i (hi_i + lo_i) v_i^T accumulates in fp32 in tensor memory without
// passing the scaled operand through shared memory. float32 caches take a
// SIMT fp32 kernel of the same contract.
#include "jacap_dev.cuh"
#include "jacap_internal.h"
#include "k_gram_body.cuh"

namespace jacap {

// ---------------------------------------------------------------- weights --
// w_i of Eq. 8 summed over the G query heads of the group (GQA heads add their
// weights): w_i = wdiv * sum_h [alpha_bar (1 - alpha_bar)]^2 kappa_h,i with
// alpha_bar = exp(l_h,i - M_h) / Z_h; with the linear surrogate (S_C = I)
// rho = 1 and w_i = wdiv * sum_h kappa_h,i. One streaming pass over the K pass's
// logits/kappa rows that writes w, for float32 caches (with bf16 caches the
// tensor-core Gram computes the same weights itself).
constexpr int WT_THREADS = 256;

template <int G>
__global__ void __launch_bounds__(WT_THREADS) weight_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  pdl_wait();
  __shared__ int s_skip;
  const int tid = threadIdx.x;
  if (tid == 0) s_skip = status_failed(ws) ? 1 : 0;
  __syncthreads();
  if (s_skip) return;
  bool bad = false, cont = false;
  float u[2 * G];
  Item item;
  for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
    if (!cont) load_unit_stats<G>(dm, ws, item.plane, item.seq, u);  // a new unit: its (M_h, 1 / Z_h)
    cont = is.next_same_unit(item);
    const int64_t base = (int64_t)item.plane * dm.Ntot;
    // four tokens per thread per round, their loads issued together
    for (int64_t t4 = item.t0 + tid; t4 < item.t1; t4 += 4 * WT_THREADS) {
      float lk[4][2 * G];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int64_t tok = t4 + q * WT_THREADS;
        const float* src = ws.lk + (base + (tok < item.t1 ? tok : t4)) * (2 * G);
        load_floats<2 * G, LkAlign<G>::ROW>(lk[q], src);
      }
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int64_t tok = t4 + q * WT_THREADS;
        if (tok >= item.t1) break;
        float wt = 0.f;
        if (dm.linear) {  // S_C = I: rho = 1
#pragma unroll
          for (int h = 0; h < G; ++h) wt += lk[q][G + h];
        } else {
#pragma unroll
          for (int h = 0; h < G; ++h) {
            const float a = expf(lk[q][h] - u[h]) * u[G + h];  // alpha_bar
            const float rho = a * (1.f - a);                    // diagonal of the softmax Jacobian
            wt = fmaf(rho * rho, lk[q][G + h], wt);             // rho^2 kappa
          }
        }
        wt *= dm.wdiv;
        bad |= !isfinite(wt);
        ws.w[base + tok] = wt;
      }
    }
  }
  if (bad) flag(ws, ST_NONFINITE);
}

template <int G>
__global__ void __launch_bounds__(GR_THREADS, 1)
    gram_bf16_kernel(const __grid_constant__ CUtensorMap vmap, Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  pdl_wait();
  gram_bf16_body<G, false>(&vmap, dm, ws, blockIdx.x, gridDim.x);
}

// ------------------------------------------------------------ SIMT fp32 ---
// float32 caches: thread t accumulates the 8x8 block (rows 8*(t/16), cols
// 8*(t%16)) of the chunk's partial Gram over 32-token slabs staged in SMEM.
constexpr int GF_THREADS = 256;
constexpr int GF_SLAB = 32;
constexpr int GF_LD = D + 4;

__global__ void __launch_bounds__(GF_THREADS)
    gram_f32_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu, const float* __restrict__ v) {
  pdl_wait();
  __shared__ __align__(16) float xs[GF_SLAB][GF_LD];  // w_i v_i (16-byte rows: GF_LD is a multiple of 4)
  __shared__ __align__(16) float vs[GF_SLAB][GF_LD];  // v_i
  __shared__ float wsl[GF_SLAB];
  __shared__ int s_skip;
  const int tid = threadIdx.x;
  if (tid == 0) s_skip = status_failed(ws) ? 1 : 0;
  __syncthreads();
  if (s_skip) return;
  const int rb = tid / 16, cb = tid % 16;
  Item item;
  for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
    const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
    const float* vbase = v + (int64_t)l * dm.kv_sl + (int64_t)g * dm.kv_sh;
    float2 acc[8][4];  // columns (2 q, 2 q + 1) of row p, packed multiply-adds
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = make_float2(0.f, 0.f);
    for (int64_t t = item.t0; t < item.t1; t += GF_SLAB) {
      if (tid < GF_SLAB) {
        const int64_t tok = t + tid;
        wsl[tid] = tok < item.t1 ? ws.w[(int64_t)item.plane * dm.Ntot + tok] : 0.f;
      }
      __syncthreads();
#pragma unroll
      for (int e = tid; e < GF_SLAB * (D / 4); e += GF_THREADS) {  // all loads in flight before the stores
        const int r = e / (D / 4), c4 = (e % (D / 4)) * 4;
        const int64_t tok = t + r;
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (tok < item.t1) x = *(const float4*)(vbase + tok * dm.kv_st + c4);
        const float wt = wsl[r];
        *(float4*)&vs[r][c4] = x;
        *(float4*)&xs[r][c4] = make_float4(wt * x.x, wt * x.y, wt * x.z, wt * x.w);
      }
      __syncthreads();
#pragma unroll 4
      for (int r = 0; r < GF_SLAB; ++r) {
        const float4 a0 = *(const float4*)&vs[r][rb * 8], a1 = *(const float4*)&vs[r][rb * 8 + 4];
        const float4 b0 = *(const float4*)&xs[r][cb * 8], b1 = *(const float4*)&xs[r][cb * 8 + 4];
        const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
        const float2 b[4] = {make_float2(b0.x, b0.y), make_float2(b0.z, b0.w), make_float2(b1.x, b1.y),
                             make_float2(b1.z, b1.w)};
#pragma unroll
        for (int p = 0; p < 8; ++p)
#pragma unroll
          for (int q = 0; q < 4; ++q) acc[p][q] = __ffma2_rn(make_float2(a[p], a[p]), b[q], acc[p][q]);
      }
      __syncthreads();
    }
    float* dst = ws.gpart + ((int64_t)item.plane * dm.c_cap + item.cidx) * D * D;
    if (tid == 0) ws.pflag[(int64_t)item.plane * dm.c_cap + item.cidx] = 1;  // a partial per chunk here
    if ((rb * 8) >> 5 < (cb * 8) >> 5) continue;  // upper 32 x 32 blocks: not read (symmetry)
#pragma unroll
    for (int p = 0; p < 8; ++p) {
      // (m, n) at ((n / 32) D + m) 32 + n % 32; the 8 columns share one block
      const int m = rb * 8 + p, n0 = cb * 8;
      float* row = dst + ((n0 >> 5) * D + m) * 32 + (n0 & 31);
      *(float4*)row = make_float4(acc[p][0].x, acc[p][0].y, acc[p][1].x, acc[p][1].y);
      *(float4*)(row + 4) = make_float4(acc[p][2].x, acc[p][2].y, acc[p][3].x, acc[p][3].y);
    }
  }
}

// ------------------------------------------------------- unit statistics --
// Warp h of block u merges the chunk statistics of unit u for query head h
// (unit_softmax_stats_warp) and stores (M_h, 1 / Z_h) in ws.ustats, so the
// weight computations read two floats per head instead of merging the unit's
// chunks themselves at every unit they start.
template <int G>
__global__ void __launch_bounds__(32 * G) unit_stats_kernel(Dims dm, Ws ws) {
  pdl_wait();
  if (status_failed(ws)) return;
  const int u = blockIdx.x, h = threadIdx.x >> 5;
  float M, Z;
  unit_softmax_stats_warp<G>(dm, ws, u / dm.S, u % dm.S, h, M, Z);
  if ((threadIdx.x & 31) == 0) {
    ws.ustats[(int64_t)u * 2 * G + h] = M;
    ws.ustats[(int64_t)u * 2 * G + G + h] = 1.f / Z;
  }
}

template <int G>
static cudaError_t launch_unit_stats_g(const Dims& dm, const Ws& ws, cudaStream_t st) {
  JACAP_TRY(launch_pdl(dm.pdl != 0, unit_stats_kernel<G>, dm.L * dm.Hkv * dm.S, 32 * G, 0, st, dm, ws));
  return cudaGetLastError();
}

cudaError_t launch_unit_stats(const Dims& dm, const Ws& ws, cudaStream_t st) {
  switch (dm.G) {
    case 1: return launch_unit_stats_g<1>(dm, ws, st);
    case 2: return launch_unit_stats_g<2>(dm, ws, st);
    case 3: return launch_unit_stats_g<3>(dm, ws, st);
    case 4: return launch_unit_stats_g<4>(dm, ws, st);
    case 5: return launch_unit_stats_g<5>(dm, ws, st);
    case 6: return launch_unit_stats_g<6>(dm, ws, st);
    case 7: return launch_unit_stats_g<7>(dm, ws, st);
    case 8: return launch_unit_stats_g<8>(dm, ws, st);
    default: return cudaErrorInvalidValue;
  }
}

// ------------------------------------------------------------ launchers ----
template <int G>
static cudaError_t launch_weights_g(const Dims& dm, const Ws& ws, const int32_t* cu, int grid, cudaStream_t st) {
  JACAP_TRY(launch_pdl(dm.pdl != 0, weight_kernel<G>, grid, WT_THREADS, 0, st, dm, ws, cu));
  return cudaGetLastError();
}

cudaError_t launch_weights(const Dims& dm, const Ws& ws, const int32_t* cu, int grid, cudaStream_t st) {
  switch (dm.G) {
    case 1: return launch_weights_g<1>(dm, ws, cu, grid, st);
    case 2: return launch_weights_g<2>(dm, ws, cu, grid, st);
    case 3: return launch_weights_g<3>(dm, ws, cu, grid, st);
    case 4: return launch_weights_g<4>(dm, ws, cu, grid, st);
    case 5: return launch_weights_g<5>(dm, ws, cu, grid, st);
    case 6: return launch_weights_g<6>(dm, ws, cu, grid, st);
    case 7: return launch_weights_g<7>(dm, ws, cu, grid, st);
    case 8: return launch_weights_g<8>(dm, ws, cu, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

template <int G>
static cudaError_t launch_gram_bf16(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, const int32_t* cu,
                                   int grid, cudaStream_t st) {
  constexpr size_t smem = GrCfg<G>::SMEM;
  cudaError_t e = cudaFuncSetAttribute(gram_bf16_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  JACAP_TRY(launch_pdl(dm.pdl != 0, gram_bf16_kernel<G>, grid, GR_THREADS, smem, st, vmap, dm, ws, cu));
  return cudaGetLastError();
}

cudaError_t launch_gram(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, int dtype, const void* v,
                        const int32_t* cu, int grid, cudaStream_t st) {
  if (dtype == 1) {
    switch (dm.G) {
      case 1: return launch_gram_bf16<1>(vmap, dm, ws, cu, grid, st);
      case 2: return launch_gram_bf16<2>(vmap, dm, ws, cu, grid, st);
      case 3: return launch_gram_bf16<3>(vmap, dm, ws, cu, grid, st);
      case 4: return launch_gram_bf16<4>(vmap, dm, ws, cu, grid, st);
      case 5: return launch_gram_bf16<5>(vmap, dm, ws, cu, grid, st);
      case 6: return launch_gram_bf16<6>(vmap, dm, ws, cu, grid, st);
      case 7: return launch_gram_bf16<7>(vmap, dm, ws, cu, grid, st);
      case 8: return launch_gram_bf16<8>(vmap, dm, ws, cu, grid, st);
      default: return cudaErrorInvalidValue;
    }
  } else {
    JACAP_TRY(launch_pdl(dm.pdl != 0, gram_f32_kernel, grid, GF_THREADS, 0, st, dm, ws, cu, (const float*)v));
  }
  return cudaGetLastError();
}

}  // namespace jacap
