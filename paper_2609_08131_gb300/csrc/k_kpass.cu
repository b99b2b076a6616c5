// k_kpass.cu - streaming K pass for bf16 caches.
//
// For every token i of a unit and every query head h of its GQA group:
//   l_h,i     = k_i . mu_h / (tau sqrt d)      pool-softmax logit (Sec. 3.4; Alg. 1 step 1)
//   kappa_h,i = sum_c lambda_h,c k_i,c^2       diagonal query-response variance (Sec. 3.4)
// plus an online (max, sum exp(l - max)) per work item and head, which the
// weight pass combines into the softmax normaliser.
//
// Both sums are 128 x 128 x N contractions per 128-token tile and run on the
// tensor cores, with fp32 accumulation in tensor memory:
//   logits: A = the TMA-staged K tile (shared memory, K-major), B = mu' =
//           mu / (tau sqrt d) split exactly into three bf16 parts (hi + mid +
//           lo carries ~24 significant bits) for the G heads;
//   kappa:  A = k^2 in tensor memory, B = lambda split the same way. A bf16
//           k has 8 significant bits, so k^2 is exact in fp32 and splits
//           exactly into hi = k^2 truncated to bf16 plus lo = k^2 - hi (at
//           most 8 significant bits, exact in bf16); two MMA chains add hi
//           and lo.
// Each thread of a compute group owns one token row (its tensor-memory lane):
// it reads the row once from shared memory, writes hi and lo of k^2 into
// tensor memory with wide stores, and reads the logits and kappa back. Three
// groups of four warps (two for G = 8) take tiles round-robin, each with its
// own k^2 buffer, so one group's MMAs run while the others build; a group
// reads a tile back only after building its next one. TMA keeps six tiles in
// flight.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int KB_STAGES = 6;
constexpr int KB_BOX = 16384;    // {64 channels, 128 tokens} bf16
constexpr int KB_TILE_BYTES = 2 * KB_BOX;
constexpr int KB_NACC = 4;       // tensor-memory result buffers
constexpr uint32_t KB_TMEM_COLS = 512;

template <int G>
struct KbCfg {
  static constexpr int NB = (3 * G <= 16) ? 16 : 32;  // MMA N = rows of each B image
  static constexpr int DC = 2 * NB;                    // result columns per buffer: logits, then kappa
  static constexpr int NG = G == 8 ? 2 : 3;            // compute groups (each 4 warps + a k^2 buffer)
  static constexpr int THREADS = 64 + 128 * NG;        // warp 0: TMA, warp 1: B images + MMA, then groups
  static constexpr uint32_t ACOL = KB_TMEM_COLS - 128 * NG;  // k^2 of group g: [ACOL + 128 g, +64) hi, [+64, +128) lo
  static_assert(KB_NACC * DC <= (int)ACOL, "tensor memory budget");
  static constexpr int IMG_ATOM = NB * 128;            // bytes per 64-channel atom
  static constexpr int IMG_BYTES = 2 * IMG_ATOM;
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, NB, 0, 0);
  static constexpr size_t SMEM = 1024 + (size_t)KB_STAGES * KB_TILE_BYTES + 4 * IMG_BYTES + 4 * NG * 2 * G * 4 + 256;
};

// B image of one item: rows n = part * G + h hold part (0 hi, 1 mid, 2 lo) of
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

// Read back the logits and kappa of own tile `pit` (token row y of the tile
// starting at `pt`), release its result buffer, write l and kappa, and fold
// the logits into the running softmax statistics. False after an abort.
template <int G>
__device__ __forceinline__ bool kb_readout(uint32_t tmem, uint32_t lanes, uint64_t* accfull, uint64_t* accempty,
                                           uint32_t pit, int64_t pt, const Item& item, int y, int lane,
                                           const Dims& dm, const Ws& ws, volatile int* abort, float (&run_m)[G],
                                           float (&run_s)[G], bool& bad) {
  using C = KbCfg<G>;
  const int ab = pit % KB_NACC;
  if (!mbar_wait(smem_u32(&accfull[ab]), (pit / KB_NACC) & 1, ws, abort)) return false;
  tc_fence_after();
  float dv[C::DC];
  const uint32_t ta = tmem + ab * C::DC + lanes;
  tmem_ld32(ta, dv);
  if constexpr (C::DC == 64) tmem_ld32(ta + 32, dv + 32);
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive(smem_u32(&accempty[ab]));
  const int64_t tok = pt + y;
  if (tok < item.t1) {
    float out[2 * G];
#pragma unroll
    for (int h = 0; h < G; ++h) {
      const float lg = dv[h] + dv[G + h] + dv[2 * G + h];
      const float kp = dv[C::NB + h] + dv[C::NB + G + h] + dv[C::NB + 2 * G + h];
      out[h] = lg;
      out[G + h] = kp;
      bad |= !isfinite(lg) || !isfinite(kp);
      if (lg > run_m[h]) {
        run_s[h] = run_s[h] * expf(run_m[h] - lg) + 1.f;
        run_m[h] = lg;
      } else {
        run_s[h] += expf(lg - run_m[h]);
      }
    }
    float* dst = ws.lk + ((int64_t)item.plane * dm.Ntot + tok) * (2 * G);
    if constexpr ((2 * G) % 4 == 0) {
#pragma unroll
      for (int e = 0; e < 2 * G; e += 4) *(float4*)(dst + e) = make_float4(out[e], out[e + 1], out[e + 2], out[e + 3]);
    } else {
#pragma unroll
      for (int e = 0; e < 2 * G; ++e) dst[e] = out[e];
    }
  }
  return true;
}

template <int G>
__global__ void __launch_bounds__(KbCfg<G>::THREADS, 1)
    kpass_bf16_kernel(const __grid_constant__ CUtensorMap kmap, Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  using C = KbCfg<G>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tiles = smem;
  uint8_t* img = tiles + KB_STAGES * KB_TILE_BYTES;  // [parity][mu, lambda][IMG_BYTES]
  float* red = (float*)(img + 4 * C::IMG_BYTES);      // [compute warps][2G]
  uint64_t* full = (uint64_t*)(red + 4 * C::NG * 2 * G);
  uint64_t* empty = full + KB_STAGES;
  uint64_t* accfull = empty + KB_STAGES;
  uint64_t* accempty = accfull + KB_NACC;
  uint64_t* afull = accempty + KB_NACC;
  uint64_t* aempty = afull + 3;
  uint64_t* imgfree = aempty + 3;
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
    for (int i = 0; i < C::NG; ++i) {
      mbar_init(smem_u32(&afull[i]), 4);
      mbar_init(smem_u32(&aempty[i]), 1);
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
    // ------------------------------------------ B images + MMA issuer -----
    uint32_t it = 0, nitem = 0;
    bool ok = true;
    Item item;
    for (int64_t i = blockIdx.x; ok && decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
      const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
      const int p = nitem & 1;
      if (nitem >= 2 && !mbar_wait(smem_u32(&imgfree[p]), ((nitem >> 1) - 1) & 1, ws, abort)) break;
      uint8_t* im_mu = img + (2 * p) * C::IMG_BYTES;
      uint8_t* im_lam = img + (2 * p + 1) * C::IMG_BYTES;
      const int64_t qb = (((int64_t)item.seq * dm.L + l) * dm.Hq + (int64_t)g * G) * D;
      build_split_image<G>(im_mu, ws.mu + qb, lane);
      build_split_image<G>(im_lam, ws.lam + qb, lane);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        tc_fence_after();
        const uint32_t ia = smem_u32(im_mu), il = smem_u32(im_lam);
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int st = it % KB_STAGES;
          const int ab = it % KB_NACC;
          const int grp = it % C::NG;
          if (!mbar_wait(smem_u32(&full[st]), (it / KB_STAGES) & 1, ws, abort) ||
              !mbar_wait(smem_u32(&afull[grp]), (it / C::NG) & 1, ws, abort) ||
              (it >= (uint32_t)KB_NACC &&
               !mbar_wait(smem_u32(&accempty[ab]), ((it / KB_NACC) & 1) ^ 1, ws, abort))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t ka = smem_u32(tiles + st * KB_TILE_BYTES);
          const uint32_t dl = tmem + ab * C::DC;  // logits
          const uint32_t dk = dl + C::NB;         // kappa: hi and lo parts of k^2 accumulate here
          const uint32_t aq = tmem + C::ACOL + 128 * grp;
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {  // 16 channels per MMA; three chains interleaved
            const uint64_t ad = smem_desc_sw128(ka + (k >> 2) * KB_BOX + (k & 3) * 32, 16, 1024);
            const uint64_t bm = smem_desc_sw128(ia + (k >> 2) * C::IMG_ATOM + (k & 3) * 32, 16, 1024);
            const uint64_t bl = smem_desc_sw128(il + (k >> 2) * C::IMG_ATOM + (k & 3) * 32, 16, 1024);
            umma_f16_ss(dl, ad, bm, C::IDESC, k > 0 ? 1u : 0u);
            umma_f16_ts(dk, aq + 8 * k, bl, C::IDESC, k > 0 ? 1u : 0u);
            umma_f16_ts(dk, aq + 64 + 8 * k, bl, C::IDESC, 1u);
          }
          umma_commit(smem_u32(&empty[st]));
          umma_commit(smem_u32(&aempty[grp]));
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
    const int grp = (warp - 2) >> 2;        // tiles with it % NG == grp
    const int quarter = warp & 3;
    const int y = quarter * 32 + lane;      // token row owned (tensor-memory lane)
    const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
    const uint32_t aq = tmem + C::ACOL + 128 * grp + lanes;
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
      // The readout of an own tile is deferred until the group has built the
      // k^2 operand of its next own tile, so the tile's MMAs run meanwhile.
      bool have = false;
      uint32_t p_it = 0;
      int64_t p_t = 0;
      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        if ((int)(it % C::NG) != grp) continue;
        const int st = it % KB_STAGES;
        if (!mbar_wait(smem_u32(&full[st]), (it / KB_STAGES) & 1, ws, abort)) goto compute_done;
        if (it >= (uint32_t)C::NG &&
            !mbar_wait(smem_u32(&aempty[grp]), ((it / C::NG) & 1) ^ 1, ws, abort))
          goto compute_done;
        tc_fence_after();
        const uint8_t* kt = tiles + st * KB_TILE_BYTES;
        // ---- k^2 = hi + lo (exact) into tensor memory, 32 channels at a time ----
#pragma unroll
        for (int cq = 0; cq < 4; ++cq) {
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const int ch = 4 * cq + j;  // 16-byte chunk: channels 8 ch .. 8 ch + 7
            const uint4 raw = *(const uint4*)(kt + (ch >> 3) * KB_BOX + sw128_off(y, ch & 7));
            const uint32_t rw[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              const float2 kk = make_float2(bf16lo(rw[q]), bf16hi(rw[q]));
              const float2 sq = __fmul2_rn(kk, kk);
              const uint32_t s0 = __float_as_uint(sq.x), s1 = __float_as_uint(sq.y);
              const float2 ht = make_float2(__uint_as_float(s0 & 0xFFFF0000u), __uint_as_float(s1 & 0xFFFF0000u));
              const float2 rr = __ffma2_rn(ht, make_float2(-1.f, -1.f), sq);
              hi[4 * j + q] = __byte_perm(s0, s1, 0x7632);
              lo[4 * j + q] = __byte_perm(__float_as_uint(rr.x), __float_as_uint(rr.y), 0x7632);
            }
          }
          tmem_st_32x32b_x16(aq + 16 * cq, hi);
          tmem_st_32x32b_x16(aq + 64 + 16 * cq, lo);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&empty[st]));
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&afull[grp]));
        if (have && !kb_readout<G>(tmem, lanes, accfull, accempty, p_it, p_t, item, y, lane, dm, ws, abort, run_m,
                                   run_s, bad))
          goto compute_done;
        have = true;
        p_it = it;
        p_t = t;
      }
      if (have && !kb_readout<G>(tmem, lanes, accfull, accempty, p_it, p_t, item, y, lane, dm, ws, abort, run_m,
                                 run_s, bad))
        goto compute_done;
      // ---- per-item softmax statistics: warp butterflies, then 8 warps ----
      const int cw = warp - 2;
#pragma unroll
      for (int h = 0; h < G; ++h) {
        softmax_warp_merge(run_m[h], run_s[h]);
        if (lane == 0) {
          red[cw * 2 * G + h] = run_m[h];
          red[cw * 2 * G + G + h] = run_s[h];
        }
      }
      named_barrier_sync(1, 128 * C::NG);
      if (tid - 64 < G) {
        const int h = tid - 64;
        float m = -INFINITY, ssum = 0.f;
        for (int j = 0; j < 4 * C::NG; ++j) softmax_merge(m, ssum, red[j * 2 * G + h], red[j * 2 * G + G + h]);
        float* cs = ws.cstats + (((int64_t)item.plane * dm.c_cap + item.cidx) * G + h) * 2;
        cs[0] = m;
        cs[1] = ssum;
      }
      named_barrier_sync(1, 128 * C::NG);
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
  kpass_bf16_kernel<G><<<grid, KbCfg<G>::THREADS, smem, st>>>(kmap, dm, ws, cu);
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
