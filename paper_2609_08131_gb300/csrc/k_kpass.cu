// k_kpass.cu - streaming K pass for bf16 caches.
//
// For every token i of a unit and every query head h of its GQA group:
//   l_h,i     = k_i . mu_h / (tau sqrt d)      pool-softmax logit (Sec. 3.4; Alg. 1 step 1)
//   kappa_h,i = sum_c lambda_h,c k_i,c^2       diagonal query-response variance (Sec. 3.4)
// plus an online (max, sum exp(l - max)) per work item and head, which the
// weight pass combines into the softmax normaliser.
//
// Layout of the work: TMA streams 128-token K tiles (128-byte swizzle) through
// a 6-stage ring. The logits are a 128 x 128 x N contraction per tile and run
// on the tensor cores: B holds mu' = mu/(tau sqrt d) split exactly into three
// bf16 parts (hi + mid + lo carries ~24 significant bits) for the G heads, and
// the fp32 result lands in tensor memory. kappa needs elementwise squares and
// runs on the CUDA cores: eight lanes share a token, each keeps its 16
// channels of lambda in registers and the G partial sums are combined with a
// reduce-scatter over the eight lanes. Two groups of four warps take
// alternate tiles; each reads back the logits of its tile from tensor memory
// (one thread per token), writes l and kappa, and keeps the online statistics.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int KB_THREADS = 320;  // warp 0: TMA, warp 1: mu image + MMA, warps 2-9: two compute groups
constexpr int KB_STAGES = 6;
constexpr int KB_BOX = 16384;    // {64 channels, 128 tokens} bf16
constexpr int KB_TILE_BYTES = 2 * KB_BOX;
constexpr int KB_NACC = 4;       // tensor-memory logit buffers
constexpr uint32_t KB_TMEM_COLS = 128;

template <int G>
struct KbCfg {
  static constexpr int NB = (3 * G <= 16) ? 16 : 32;  // MMA N = rows of the mu image
  static constexpr int IMG_ATOM = NB * 128;            // bytes per 64-channel atom
  static constexpr int IMG_BYTES = 2 * IMG_ATOM;
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, NB, 0, 0);
  static constexpr size_t SMEM = 1024 + (size_t)KB_STAGES * KB_TILE_BYTES + 2 * IMG_BYTES +
                                 (size_t)2 * 128 * 2 * G * 4 + 256;
};

template <int G>
__global__ void __launch_bounds__(KB_THREADS, 1)
    kpass_bf16_kernel(const __grid_constant__ CUtensorMap kmap, Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  using C = KbCfg<G>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tiles = smem;
  uint8_t* img = tiles + KB_STAGES * KB_TILE_BYTES;                  // [2][IMG_BYTES]
  float* red = (float*)(img + 2 * C::IMG_BYTES);                      // [2 groups][128][2G]
  uint64_t* full = (uint64_t*)(red + 2 * 128 * 2 * G);
  uint64_t* empty = full + KB_STAGES;
  uint64_t* accfull = empty + KB_STAGES;
  uint64_t* accempty = accfull + KB_NACC;
  uint64_t* imgfree = accempty + KB_NACC;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_skip;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_abort = 0;
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < KB_STAGES; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 5);  // MMA commit + the 4 warps of the group that owns the tile
    }
    for (int i = 0; i < KB_NACC; ++i) {
      mbar_init(smem_u32(&accfull[i]), 1);
      mbar_init(smem_u32(&accempty[i]), 4);
    }
    mbar_init(smem_u32(&imgfree[0]), 1);
    mbar_init(smem_u32(&imgfree[1]), 1);
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
    // ------------------------------------ mu image builder + MMA issuer ---
    uint32_t it = 0, nitem = 0;
    bool ok = true;
    Item item;
    for (int64_t i = blockIdx.x; ok && decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
      const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
      const int p = nitem & 1;
      if (nitem >= 2 && !mbar_wait(smem_u32(&imgfree[p]), ((nitem >> 1) - 1) & 1, ws, abort)) break;
      // B image rows n = part * G + h (part 0/1/2 = hi/mid/lo of mu'_h), K-major, 128-byte swizzle
      uint8_t* im = img + p * C::IMG_BYTES;
      const float* mu = ws.mu + (((int64_t)item.seq * dm.L + l) * dm.Hq + (int64_t)g * G) * D;
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
              const float v = mu[h * D + cc * 8 + 2 * q + z];
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
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        tc_fence_after();
        const uint32_t ia = smem_u32(im);
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
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {  // 16 channels per MMA
            const uint64_t ad = smem_desc_sw128(ka + (k >> 2) * KB_BOX + (k & 3) * 32, 16, 1024);
            const uint64_t bd = smem_desc_sw128(ia + (k >> 2) * C::IMG_ATOM + (k & 3) * 32, 16, 1024);
            umma_f16_ss(tmem + ab * 32, ad, bd, C::IDESC, k > 0 ? 1u : 0u);
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
  } else {
    // ---------------------------------------------- compute groups --------
    const int grp = (warp - 2) >> 2;        // tiles with it % 2 == grp
    const int wg = (warp - 2) & 3;          // warp index within the group == TMEM lane quarter
    const int quarter = warp & 3;
    const int y = quarter * 32 + lane;      // token row owned for the logits (TMEM lane)
    const int sub = lane & 7;               // kappa: lane within the 8-lane token group
    const int tg = wg * 4 + (lane >> 3);    // kappa: token group 0..15 of the group
    const int gidx = tid - 64;              // 0..255 across both groups
    uint32_t it = 0;
    bool bad = false;
    Item item;
    for (int64_t i = blockIdx.x; decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
      const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
      // lambda of this lane's 16 channels (8 sub..8 sub+7 and 64+8 sub..), all heads
      float lam[G][16];
      {
        const float* lp = ws.lam + (((int64_t)item.seq * dm.L + l) * dm.Hq + (int64_t)g * G) * D;
#pragma unroll
        for (int h = 0; h < G; ++h) {
#pragma unroll
          for (int q = 0; q < 8; q += 4) {
            const float4 a = *(const float4*)(lp + h * D + 8 * sub + q);
            const float4 b = *(const float4*)(lp + h * D + 64 + 8 * sub + q);
            lam[h][q] = a.x; lam[h][q + 1] = a.y; lam[h][q + 2] = a.z; lam[h][q + 3] = a.w;
            lam[h][8 + q] = b.x; lam[h][8 + q + 1] = b.y; lam[h][8 + q + 2] = b.z; lam[h][8 + q + 3] = b.w;
          }
        }
      }
      float run_m[G], run_s[G];
#pragma unroll
      for (int h = 0; h < G; ++h) {
        run_m[h] = -INFINITY;
        run_s[h] = 0.f;
      }
      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        if ((int)(it & 1) != grp) continue;
        const int st = it % KB_STAGES;
        const int ab = it % KB_NACC;
        if (!mbar_wait(smem_u32(&full[st]), (it / KB_STAGES) & 1, ws, abort)) goto compute_done;
        const uint8_t* kt = tiles + st * KB_TILE_BYTES;
        // ---- kappa: 8 steps of 16 tokens, 8 lanes per token ----
        uint4 rr[16];  // this lane's two 16-byte chunks of its token row, all 8 steps
#pragma unroll
        for (int s8 = 0; s8 < 8; ++s8) {
          const int yk = 16 * s8 + tg;
          rr[2 * s8] = *(const uint4*)(kt + sw128_off(yk, sub));
          rr[2 * s8 + 1] = *(const uint4*)(kt + KB_BOX + sw128_off(yk, sub));
        }
#pragma unroll
        for (int s8 = 0; s8 < 8; ++s8) {
          const int yk = 16 * s8 + tg;
          const uint32_t rw[8] = {rr[2 * s8].x, rr[2 * s8].y, rr[2 * s8].z, rr[2 * s8].w,
                                  rr[2 * s8 + 1].x, rr[2 * s8 + 1].y, rr[2 * s8 + 1].z, rr[2 * s8 + 1].w};
          float2 acc[G];
#pragma unroll
          for (int h = 0; h < G; ++h) acc[h] = make_float2(0.f, 0.f);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const float2 kk = make_float2(bf16lo(rw[q]), bf16hi(rw[q]));
            const float2 sq = __fmul2_rn(kk, kk);
#pragma unroll
            for (int h = 0; h < G; ++h) acc[h] = __ffma2_rn(sq, make_float2(lam[h][2 * q], lam[h][2 * q + 1]), acc[h]);
          }
          float v[G];
#pragma unroll
          for (int h = 0; h < G; ++h) v[h] = acc[h].x + acc[h].y;
          // reduce-scatter of the G sums over the 8 lanes of the token group
          int base = 0;  // first head index this lane still holds
#pragma unroll
          for (int span = G, bit = 4; bit >= 1; bit >>= 1) {
            if (span > 1) {
              const int halfspan = span >> 1;
              const bool upper = (sub & bit) != 0;
#pragma unroll
              for (int j = 0; j < halfspan; ++j) {
                const float send = upper ? v[j] : v[halfspan + j];
                const float recv = __shfl_xor_sync(0xffffffffu, send, bit);
                v[j] = (upper ? v[halfspan + j] : v[j]) + recv;
              }
              if (upper) base += halfspan;
              span = halfspan;
            } else {
              v[0] += __shfl_xor_sync(0xffffffffu, v[0], bit);
            }
          }
          // lanes that end with the same head hold equal sums; the lowest writes
          const int64_t tokk = t + yk;
          constexpr int REP = G >= 8 ? 1 : 8 / G;  // lanes per finished head
          if (tokk < item.t1 && (sub % REP) == 0) {
            ws.lk[((int64_t)item.plane * dm.Ntot + tokk) * (2 * G) + G + base] = v[0];
            bad |= !isfinite(v[0]);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&empty[st]));
        // ---- logits from tensor memory: one thread per token ----
        if (!mbar_wait(smem_u32(&accfull[ab]), (it / KB_NACC) & 1, ws, abort)) goto compute_done;
        tc_fence_after();
        float dv[C::NB];
        const uint32_t ta = tmem + ab * 32 + ((uint32_t)(quarter * 32) << 16);
        if constexpr (C::NB == 16) tmem_ld16(ta, dv); else tmem_ld32(ta, dv);
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
          float* dst = ws.lk + ((int64_t)item.plane * dm.Ntot + tok) * (2 * G);
          if constexpr (G % 4 == 0) {
#pragma unroll
            for (int h = 0; h < G; h += 4) *(float4*)(dst + h) = make_float4(lg[h], lg[h + 1], lg[h + 2], lg[h + 3]);
          } else {
#pragma unroll
            for (int h = 0; h < G; ++h) dst[h] = lg[h];
          }
        }
      }
      // ---- per-item softmax statistics: warp butterflies, then 8 warps ----
#pragma unroll
      for (int h = 0; h < G; ++h) {
        softmax_warp_merge(run_m[h], run_s[h]);
        if (lane == 0) {
          red[(gidx >> 5) * 2 * G + h] = run_m[h];
          red[(gidx >> 5) * 2 * G + G + h] = run_s[h];
        }
      }
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if (gidx < G) {
        const int h = gidx;
        float m = -INFINITY, ssum = 0.f;
        for (int j = 0; j < 8; ++j) softmax_merge(m, ssum, red[j * 2 * G + h], red[j * 2 * G + G + h]);
        float* cs = ws.cstats + (((int64_t)item.plane * dm.c_cap + item.cidx) * G + h) * 2;
        cs[0] = m;
        cs[1] = ssum;
      }
      asm volatile("bar.sync 1, 256;" ::: "memory");
    }
  compute_done:
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
