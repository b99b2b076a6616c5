// k_kpass.cu - streaming K pass for bf16 caches.
//
// For every token i of a unit and every query head h of its GQA group:
//   l_h,i     = k_i . mu_h / (tau sqrt d)      pool-softmax logit (Sec. 3.4; Alg. 1 step 1)
//   kappa_h,i = sum_c lambda_h,c k_i,c^2       diagonal query-response variance (Sec. 3.4)
// plus an online (max, sum exp(l - max)) per work item and head, which the
// weight pass combines into the softmax normaliser.
//
// The logits are a 128 x 128 x N contraction per 128-token tile and run on the
// tensor cores: A = the TMA-staged K tile (shared memory, K-major), B = mu' =
// mu / (tau sqrt d) split exactly into three bf16 parts (hi + mid + lo carries
// ~24 significant bits) for the G heads, fp32 accumulation in tensor memory.
// kappa needs the elementwise squares of k, which would double the tensor
// instructions (k^2 has 16 significant bits: two bf16 operands) at a fixed
// cost per instruction, so it runs on the CUDA cores instead: k^2 is exact in
// fp32 and is weighted by lambda (fp32, broadcast from shared memory) with
// packed fp32x2 multiply-adds.
//
// Warp roles: 0 TMA producer (six tiles in flight); 1 builds the mu' image
// and lambda of each item and issues the logits MMAs; 2-5 kappa (a pair of
// warps per tile, two tokens per lane, the pairs alternate tiles); 6-9 read the
// logits back from tensor memory (one lane quarter each) and keep the online
// softmax statistics.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int KB_STAGES = 6;
constexpr int KB_BOX = 16384;    // {64 channels, 128 tokens} bf16
constexpr int KB_TILE_BYTES = 2 * KB_BOX;
constexpr int KB_NACC = 4;       // tensor-memory logits buffers
constexpr uint32_t KB_TMEM_COLS = 128;
constexpr int KB_THREADS = 320;
constexpr int KB_KAPPA_WARP0 = 2, KB_READ_WARP0 = 6;

template <int G>
struct KbCfg {
  static constexpr int NB = (3 * G <= 16) ? 16 : 32;  // MMA N = rows of the mu' image
  static constexpr int IMG_ATOM = NB * 128;            // bytes per 64-channel atom
  static constexpr int IMG_BYTES = 2 * IMG_ATOM;
  static constexpr int LAM_BYTES = G * D * 4;          // lambda, fp32 [G][128]
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, NB, 0, 0);
  static_assert(KB_NACC * NB <= (int)KB_TMEM_COLS, "tensor memory budget");
  static constexpr size_t SMEM =
      1024 + (size_t)KB_STAGES * KB_TILE_BYTES + 2 * IMG_BYTES + 2 * LAM_BYTES + 4 * 2 * G * 4 + 512;
};

// mu' image of one item: rows n = part * G + h hold part (0 hi, 1 mid, 2 lo) of
// src[h][0..127], K-major with the 128-byte swizzle (two 64-channel atoms).
template <int G>
__device__ __forceinline__ void build_split_image(uint8_t* im, const float* src, int lane) {
  using C = KbCfg<G>;
  for (int e = lane; e < C::NB * 16; e += 32) {
    const int n = e >> 4, cc = e & 15;
    uint32_t wv[4] = {0u, 0u, 0u, 0u};
    if (n < 3 * G) {
      const int part = n / G, h = n % G;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float x[2];
#pragma unroll
        for (int z = 0; z < 2; ++z) {
          const float v = src[h * D + cc * 8 + 2 * q + z];
          const float hi = __bfloat162float(__float2bfloat16_rn(v));
          const float r1 = v - hi;
          const float mid = __bfloat162float(__float2bfloat16_rn(r1));
          x[z] = part == 0 ? hi : (part == 1 ? mid : r1 - mid);
        }
        wv[q] = pack_bf16x2(x[0], x[1]);
      }
    }
    *(uint4*)(im + (cc >> 3) * C::IMG_ATOM + sw128_off(n, cc & 7)) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  }
}

// kappa of two token rows (ya, yb) of a staged tile: sum over the 16 chunks of
// 8 channels of lambda_h,c k_c^2, two independent fp32x2 chains per token and
// head.
template <int G>
__device__ __forceinline__ void kappa_two_rows(const uint8_t* kt, const float* lam, int ya, int yb, float (&ka)[G],
                                               float (&kb)[G]) {
  float2 aa[G][2], ab[G][2];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    aa[h][0] = aa[h][1] = ab[h][0] = ab[h][1] = make_float2(0.f, 0.f);
  }
#pragma unroll 2
  for (int cc = 0; cc < 16; ++cc) {
    const uint4 ra = *(const uint4*)(kt + (cc >> 3) * KB_BOX + sw128_off(ya, cc & 7));
    const uint4 rb = *(const uint4*)(kt + (cc >> 3) * KB_BOX + sw128_off(yb, cc & 7));
    const uint32_t wa[4] = {ra.x, ra.y, ra.z, ra.w}, wb[4] = {rb.x, rb.y, rb.z, rb.w};
    float2 sa[4], sb[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 xa = make_float2(bf16lo(wa[q]), bf16hi(wa[q]));
      const float2 xb = make_float2(bf16lo(wb[q]), bf16hi(wb[q]));
      sa[q] = __fmul2_rn(xa, xa);  // exact: 8-bit significands
      sb[q] = __fmul2_rn(xb, xb);
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
      const float4 l0 = *(const float4*)(lam + h * D + 8 * cc);
      const float4 l1 = *(const float4*)(lam + h * D + 8 * cc + 4);
      const float2 p0 = make_float2(l0.x, l0.y), p1 = make_float2(l0.z, l0.w);
      const float2 p2 = make_float2(l1.x, l1.y), p3 = make_float2(l1.z, l1.w);
      aa[h][0] = __ffma2_rn(sa[0], p0, aa[h][0]);
      aa[h][1] = __ffma2_rn(sa[1], p1, aa[h][1]);
      ab[h][0] = __ffma2_rn(sb[0], p0, ab[h][0]);
      ab[h][1] = __ffma2_rn(sb[1], p1, ab[h][1]);
      aa[h][0] = __ffma2_rn(sa[2], p2, aa[h][0]);
      aa[h][1] = __ffma2_rn(sa[3], p3, aa[h][1]);
      ab[h][0] = __ffma2_rn(sb[2], p2, ab[h][0]);
      ab[h][1] = __ffma2_rn(sb[3], p3, ab[h][1]);
    }
  }
#pragma unroll
  for (int h = 0; h < G; ++h) {
    ka[h] = (aa[h][0].x + aa[h][1].x) + (aa[h][0].y + aa[h][1].y);
    kb[h] = (ab[h][0].x + ab[h][1].x) + (ab[h][0].y + ab[h][1].y);
  }
}

template <int G>
__device__ __forceinline__ void store_part(float* dst, const float (&v)[G]) {
  if constexpr (G % 4 == 0) {
#pragma unroll
    for (int h = 0; h < G; h += 4) *(float4*)(dst + h) = make_float4(v[h], v[h + 1], v[h + 2], v[h + 3]);
  } else if constexpr (G == 2) {
    *(float2*)dst = make_float2(v[0], v[1]);
  } else {
    dst[0] = v[0];
  }
}

template <int G>
__global__ void __launch_bounds__(KB_THREADS, 1)
    kpass_bf16_kernel(const __grid_constant__ CUtensorMap kmap, Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  using C = KbCfg<G>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tiles = smem;
  uint8_t* img = tiles + KB_STAGES * KB_TILE_BYTES;    // [parity][IMG_BYTES] mu' images
  float* lams = (float*)(img + 2 * C::IMG_BYTES);       // [parity][G][128] lambda
  float* red = lams + 2 * G * D;                         // [4 readout warps][2G]
  uint64_t* full = (uint64_t*)(red + 4 * 2 * G);
  uint64_t* empty = full + KB_STAGES;
  uint64_t* accfull = empty + KB_STAGES;
  uint64_t* accempty = accfull + KB_NACC;
  uint64_t* imgready = accempty + KB_NACC;
  uint64_t* imgfree = imgready + 2;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_skip;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_abort = 0;
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < KB_STAGES; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 3);  // MMA commit + the two kappa warps of the tile
    }
    for (int i = 0; i < KB_NACC; ++i) {
      mbar_init(smem_u32(&accfull[i]), 1);
      mbar_init(smem_u32(&accempty[i]), 4);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&imgready[i]), 1);
      mbar_init(smem_u32(&imgfree[i]), 5);  // MMA commit + the four kappa warps
    }
    fence_mbar_init();
  }
  __syncthreads();
  if (s_skip) return;
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), KB_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  volatile int* abort = &s_abort;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer --------
    if (lane == 0) {
      prefetch_tmap(&kmap);
      uint32_t it = 0;
      bool ok = true;
      Item item;
      for (int64_t i = blockIdx.x; ok && decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        for (int64_t t = item.t0; t < item.t1; t += TILE) {
          const int st = it % KB_STAGES;
          if (it >= (uint32_t)KB_STAGES &&
              !mbar_wait(smem_u32(&empty[st]), ((it / KB_STAGES) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          uint8_t* kt = tiles + st * KB_TILE_BYTES;
          mbar_arrive_expect_tx(smem_u32(&full[st]), KB_TILE_BYTES);
          tma_load_4d(smem_u32(kt), &kmap, 0, (int)t, g, l, smem_u32(&full[st]));
          tma_load_4d(smem_u32(kt + KB_BOX), &kmap, 64, (int)t, g, l, smem_u32(&full[st]));
          ++it;
        }
      }
      for (uint32_t k = (it > (uint32_t)KB_STAGES ? it - KB_STAGES : 0); k < it; ++k)
        mbar_wait(smem_u32(&full[k % KB_STAGES]), (k / KB_STAGES) & 1, ws, nullptr);
    }
  } else if (warp == 1) {
    // ------------------------------- mu' image, lambda, logits MMA issuer --
    uint32_t it = 0, nitem = 0;
    bool ok = true;
    Item item;
    for (int64_t i = blockIdx.x; ok && decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
      const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
      const int p = nitem & 1;
      if (nitem >= 2 && !mbar_wait(smem_u32(&imgfree[p]), ((nitem >> 1) - 1) & 1, ws, abort)) break;
      uint8_t* im_mu = img + p * C::IMG_BYTES;
      float* lam_s = lams + p * G * D;
      const int64_t qb = (((int64_t)item.seq * dm.L + l) * dm.Hq + (int64_t)g * G) * D;
      build_split_image<G>(im_mu, ws.mu + qb, lane);
      for (int e = lane; e < G * D / 4; e += 32) ((float4*)lam_s)[e] = ((const float4*)(ws.lam + qb))[e];
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(smem_u32(&imgready[p]));
        tc_fence_after();
        const uint32_t ia = smem_u32(im_mu);
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int st = it % KB_STAGES;
          const int ab = it % KB_NACC;
          if (!mbar_wait(smem_u32(&full[st]), (it / KB_STAGES) & 1, ws, abort) ||
              (it >= (uint32_t)KB_NACC &&
               !mbar_wait(smem_u32(&accempty[ab]), ((it / KB_NACC) & 1) ^ 1, ws, abort))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t ka = smem_u32(tiles + st * KB_TILE_BYTES);
          const uint32_t dl = tmem + ab * C::NB;
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {  // 16 channels per MMA
            const uint64_t ad = smem_desc_sw128(ka + (k >> 2) * KB_BOX + (k & 3) * 32, 16, 1024);
            const uint64_t bm = smem_desc_sw128(ia + (k >> 2) * C::IMG_ATOM + (k & 3) * 32, 16, 1024);
            umma_f16_ss(dl, ad, bm, C::IDESC, k > 0 ? 1u : 0u);
          }
          umma_commit(smem_u32(&empty[st]));
          umma_commit(smem_u32(&accfull[ab]));
        }
        if (ok) umma_commit(smem_u32(&imgfree[p]));
      }
      it = __shfl_sync(0xffffffffu, it, 0);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      ++nitem;
    }
    // every MMA issued here completes before the CTA tears down tensor memory
    if (lane == 0 && it > 0)
      mbar_wait(smem_u32(&accfull[(it - 1) % KB_NACC]), ((it - 1) / KB_NACC) & 1, ws, nullptr);
  } else if (warp < KB_READ_WARP0) {
    // ------------------------------------------------------ kappa ---------
    const int kw = warp - KB_KAPPA_WARP0;
    const int pair = kw >> 1;                 // tiles with it % 2 == pair
    const int ya = 64 * (kw & 1) + lane;      // token rows ya and ya + 32 of the tile
    const int yb = ya + 32;
    uint32_t it = 0, nitem = 0;
    bool bad = false;
    Item item;
    for (int64_t i = blockIdx.x; decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
      const int p = nitem & 1;
      if (!mbar_wait(smem_u32(&imgready[p]), (nitem >> 1) & 1, ws, abort)) goto kappa_done;
      {
        const float* lam_s = lams + p * G * D;
        float* lkp = ws.lk + (int64_t)item.plane * dm.Ntot * (2 * G) + G;
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          if ((int)(it & 1) != pair) continue;
          const int st = it % KB_STAGES;
          if (!mbar_wait(smem_u32(&full[st]), (it / KB_STAGES) & 1, ws, abort)) goto kappa_done;
          float ka[G], kb[G];
          kappa_two_rows<G>(tiles + st * KB_TILE_BYTES, lam_s, ya, yb, ka, kb);
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&empty[st]));
#pragma unroll
          for (int h = 0; h < G; ++h) bad |= !isfinite(ka[h]) || !isfinite(kb[h]);
          if (t + ya < item.t1) store_part<G>(lkp + (t + ya) * (2 * G), ka);
          if (t + yb < item.t1) store_part<G>(lkp + (t + yb) * (2 * G), kb);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&imgfree[p]));
      ++nitem;
    }
  kappa_done:
    if (bad) flag(ws, ST_NONFINITE);
  } else {
    // ------------------------------------------ logits readout + stats ----
    const int quarter = warp & 3;
    const int y = quarter * 32 + lane;        // token row (tensor-memory lane)
    const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
    const int rw = warp - KB_READ_WARP0;
    uint32_t it = 0;
    bool bad = false;
    Item item;
    for (int64_t i = blockIdx.x; decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
      float run_m[G], run_s[G];
#pragma unroll
      for (int h = 0; h < G; ++h) {
        run_m[h] = -INFINITY;
        run_s[h] = 0.f;
      }
      float* lkp = ws.lk + (int64_t)item.plane * dm.Ntot * (2 * G);
      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        const int ab = it % KB_NACC;
        if (!mbar_wait(smem_u32(&accfull[ab]), (it / KB_NACC) & 1, ws, abort)) goto read_done;
        tc_fence_after();
        float dv[C::NB];
        if constexpr (C::NB == 16) tmem_ld16(tmem + ab * C::NB + lanes, dv);
        else tmem_ld32(tmem + ab * C::NB + lanes, dv);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&accempty[ab]));
        const int64_t tok = t + y;
        if (tok < item.t1) {
          float lg[G];
#pragma unroll
          for (int h = 0; h < G; ++h) {
            lg[h] = dv[h] + dv[G + h] + dv[2 * G + h];
            bad |= !isfinite(lg[h]);
            if (lg[h] > run_m[h]) {
              run_s[h] = run_s[h] * expf(run_m[h] - lg[h]) + 1.f;
              run_m[h] = lg[h];
            } else {
              run_s[h] += expf(lg[h] - run_m[h]);
            }
          }
          store_part<G>(lkp + tok * (2 * G), lg);
        }
      }
      // ---- per-item softmax statistics: warp butterflies, then 4 warps ----
#pragma unroll
      for (int h = 0; h < G; ++h) {
        softmax_warp_merge(run_m[h], run_s[h]);
        if (lane == 0) {
          red[rw * 2 * G + h] = run_m[h];
          red[rw * 2 * G + G + h] = run_s[h];
        }
      }
      named_barrier_sync(1, 128);
      if (rw == 0 && lane < G) {
        const int h = lane;
        float m = -INFINITY, ssum = 0.f;
        for (int j = 0; j < 4; ++j) softmax_merge(m, ssum, red[j * 2 * G + h], red[j * 2 * G + G + h]);
        float* cs = ws.cstats + (((int64_t)item.plane * dm.c_cap + item.cidx) * G + h) * 2;
        cs[0] = m;
        cs[1] = ssum;
      }
      named_barrier_sync(1, 128);
    }
  read_done:
    if (bad) flag(ws, ST_NONFINITE);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, KB_TMEM_COLS);
  }
}

template <int G>
static cudaError_t launch_g(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, const int32_t* cu, int grid,
                            cudaStream_t st) {
  constexpr size_t smem = KbCfg<G>::SMEM;
  static_assert(smem <= 232448, "shared memory budget");
  cudaError_t e = cudaFuncSetAttribute(kpass_bf16_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kpass_bf16_kernel<G><<<grid, KB_THREADS, smem, st>>>(kmap, dm, ws, cu);
  return cudaGetLastError();
}

cudaError_t launch_kpass_bf16(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, const int32_t* cu, int grid,
                              cudaStream_t st) {
  switch (dm.G) {
    case 1: return launch_g<1>(kmap, dm, ws, cu, grid, st);
    case 2: return launch_g<2>(kmap, dm, ws, cu, grid, st);
    case 4: return launch_g<4>(kmap, dm, ws, cu, grid, st);
    case 8: return launch_g<8>(kmap, dm, ws, cu, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace jacap
