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
// Warp roles: 0 TMA producer; 1 issues the logits MMAs; 14 builds the mu'
// image and lambda of each unit a CTA reaches (double-buffered, one run of the
// unit's consecutive items ahead); 2-9 kappa (two groups of four warps alternate
// tiles; in a group each warp takes one quarter of the channels for all 128
// tokens, four per lane, so every lambda value read from shared memory serves
// four tokens, and writes its partial sums of all four token subsets into the
// group's slot); 10-13 read the logits back from tensor memory (one lane
// quarter each), add the four partial kappa of their 32 tokens from the slot,
// keep the online softmax statistics and store each token's row (logits,
// kappa) in one piece. Each group has two slots (one for G > 4), handed over
// with mbarriers, so a group writes one while the readout warps read the other.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int KB_BOX = 16384;    // {64 channels, 128 tokens} bf16
constexpr int KB_TILE_BYTES = 2 * KB_BOX;
constexpr int KB_NACC = 4;       // tensor-memory logits buffers
constexpr uint32_t KB_TMEM_COLS = 128;
constexpr int KB_THREADS = 480;
constexpr int KB_KAPPA_WARP0 = 2, KB_READ_WARP0 = 10, KB_BUILD_WARP = 14;

template <int G>
struct KbCfg {
  static constexpr int NB = (3 * G <= 16) ? 16 : 32;  // MMA N = rows of the mu' image
  static constexpr int IMG_ATOM = NB * 128;            // bytes per 64-channel atom
  static constexpr int IMG_BYTES = 2 * IMG_ATOM;
  static constexpr int LAM_BYTES = G * D * 4;          // lambda, fp32 [G][128]
  // partial-kappa slots per group: two (the group writes one while the readout
  // warps read the other) when they fit beside five K stages, else one
  static constexpr int SLOTS = G <= 4 ? 2 : 1;
  static constexpr int SLOT_FLOATS = 4 * 4 * G * 32;                 // [token subset][writer][G][32]
  static constexpr int KRED_FLOATS = 2 * SLOTS * SLOT_FLOATS;        // [group][slot]
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, NB, 0, 0);
  static_assert(KB_NACC * NB <= (int)KB_TMEM_COLS, "tensor memory budget");
  static constexpr size_t smem_for(int stages) {
    return 1024 + (size_t)stages * KB_TILE_BYTES + 2 * IMG_BYTES + 2 * LAM_BYTES + KRED_FLOATS * 4 + 4 * 2 * G * 4 +
           512;
  }
  static constexpr int STAGES = smem_for(6) <= 232448 ? 6 : (smem_for(5) <= 232448 ? 5 : 4);  // K tiles in flight
  static constexpr size_t SMEM = smem_for(STAGES);
};

// The K tile `it` lands on barrier full[kb_full(it)], one per (tile parity,
// stage). A kappa group takes every other tile, so with an odd number of
// stages it sees only every other use of a stage; on a barrier per stage its
// parity wait could not tell "my tile landed" from "the other group's tile in
// this stage has not landed yet". Per (parity, stage) every waiter sees
// consecutive phases: the tile's use of its barrier is it / kb_full_period.
template <int STAGES>
__device__ __forceinline__ int kb_full(uint32_t it) { return (int)(it & 1) * STAGES + (int)(it % STAGES); }
template <int STAGES>
__device__ __forceinline__ uint32_t kb_full_parity(uint32_t it) {
  return (it / (STAGES % 2 == 0 ? STAGES : 2 * STAGES)) & 1;
}

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

// Partial kappa over channel quarter `cq` (chunks 4 cq .. 4 cq + 3 of 8
// channels) for the four token rows lane + 32 j of a staged tile:
// part[j][h] = sum_c lambda_h,c k_c^2. Each lambda load feeds JB tokens: all
// four for G = 1, 2, 4; for other groups two passes over the quarter take two
// tokens each, which halves the accumulators held at once (and keeps them in
// registers).
template <int G>
__device__ __forceinline__ void kappa_quarter(uint32_t kt, uint32_t lam, int lane, int cq, float (&part)[4][G]) {
  constexpr int JB = (G <= 2 || G == 4) ? 4 : 2;
#pragma unroll
  for (int j0 = 0; j0 < 4; j0 += JB) {
    float2 acc[JB][G];
#pragma unroll
    for (int j = 0; j < JB; ++j)
#pragma unroll
      for (int h = 0; h < G; ++h) acc[j][h] = make_float2(0.f, 0.f);
#pragma unroll 1
    for (int cc = 4 * cq; cc < 4 * cq + 4; ++cc) {
      float4 l0[G], l1[G];
#pragma unroll
      for (int h = 0; h < G; ++h) {
        l0[h] = lds_f128(lam + (h * D + 8 * cc) * 4);
        l1[h] = lds_f128(lam + (h * D + 8 * cc + 4) * 4);
      }
#pragma unroll
      for (int j = 0; j < JB; ++j) {
        const uint4 r = lds_u128(kt + (cc >> 3) * KB_BOX + sw128_off(lane + 32 * (j0 + j), cc & 7));
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
        float2 sq[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float2 x = make_float2(bf16lo(w[q]), bf16hi(w[q]));
          sq[q] = __fmul2_rn(x, x);  // exact: 8-bit significands
        }
#pragma unroll
        for (int h = 0; h < G; ++h) {
          acc[j][h] = __ffma2_rn(sq[0], make_float2(l0[h].x, l0[h].y), acc[j][h]);
          acc[j][h] = __ffma2_rn(sq[1], make_float2(l0[h].z, l0[h].w), acc[j][h]);
          acc[j][h] = __ffma2_rn(sq[2], make_float2(l1[h].x, l1[h].y), acc[j][h]);
          acc[j][h] = __ffma2_rn(sq[3], make_float2(l1[h].z, l1[h].w), acc[j][h]);
        }
      }
    }
#pragma unroll
    for (int j = 0; j < JB; ++j)
#pragma unroll
      for (int h = 0; h < G; ++h) part[j0 + j][h] = acc[j][h].x + acc[j][h].y;
  }
}

template <int G>
__global__ void __launch_bounds__(KB_THREADS, 1)
    kpass_bf16_kernel(const __grid_constant__ CUtensorMap kmap, Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  pdl_wait();
  using C = KbCfg<G>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  constexpr int KB_STAGES = C::STAGES;
  uint8_t* tiles = smem;
  uint8_t* img = tiles + KB_STAGES * KB_TILE_BYTES;    // [parity][IMG_BYTES] mu' images
  float* lams = (float*)(img + 2 * C::IMG_BYTES);       // [parity][G][128] lambda
  float* kred = lams + 2 * G * D;                        // partial kappa of the upper channel half
  float* red = kred + C::KRED_FLOATS;                    // [4 readout warps][2G]
  uint64_t* full = (uint64_t*)(red + 4 * 2 * G);  // [tile parity][stage], see kb_full
  uint64_t* empty = full + 2 * KB_STAGES;
  uint64_t* accfull = empty + KB_STAGES;
  uint64_t* accempty = accfull + KB_NACC;
  uint64_t* imgready = accempty + KB_NACC;
  uint64_t* imgfree = imgready + 2;
  uint64_t* kready = imgfree + 2;            // [group][slot] a tile's partial kappa are in the slot
  uint64_t* kfree = kready + 2 * C::SLOTS;   // [group][slot] the readout warps have read them
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_skip;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_abort = 0;
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < KB_STAGES; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&full[KB_STAGES + i]), 1);
      mbar_init(smem_u32(&empty[i]), 5);  // MMA commit + the four kappa warps of the tile
    }
    for (int i = 0; i < KB_NACC; ++i) {
      mbar_init(smem_u32(&accfull[i]), 1);
      mbar_init(smem_u32(&accempty[i]), 4);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&imgready[i]), 1);
      mbar_init(smem_u32(&imgfree[i]), 9);  // MMA commit + the eight kappa warps

    }
    for (int i = 0; i < 2 * C::SLOTS; ++i) {
      mbar_init(smem_u32(&kready[i]), 4);  // the group's four kappa warps
      mbar_init(smem_u32(&kfree[i]), 4);   // the four readout warps
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
      // time accounting (trace builds): 0 waits for a free stage, 1 the whole loop
      TRC_DECL(TR_CTA_SLOTS);
      TRC_T(tr_all);
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        for (int64_t t = item.t0; t < item.t1; t += TILE) {
          const int st = it % KB_STAGES;
          TRC_T(tr_w);
          if (it >= (uint32_t)KB_STAGES &&
              !mbar_wait(smem_u32(&empty[st]), ((it / KB_STAGES) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          TRC_ADD(0, tr_w);
          uint8_t* kt = tiles + st * KB_TILE_BYTES;
          const uint32_t fb = smem_u32(&full[kb_full<KB_STAGES>(it)]);
          mbar_arrive_expect_tx(fb, KB_TILE_BYTES);
          tma_load_4d(smem_u32(kt), &kmap, 0, (int)t, g, l, fb);
          tma_load_4d(smem_u32(kt + KB_BOX), &kmap, 64, (int)t, g, l, fb);
          ++it;
        }
      }
      TRC_ADD(1, tr_all);
      TRC_PUT(ws, TR_K_KPASS, 2);
      for (uint32_t k = (it > (uint32_t)KB_STAGES ? it - KB_STAGES : 0); k < it; ++k)
        mbar_wait(smem_u32(&full[kb_full<KB_STAGES>(k)]), kb_full_parity<KB_STAGES>(k), ws, nullptr);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ logits MMA issuer ---
    if (lane == 0) {
      uint32_t it = 0, nrun = 0;  // nrun: runs of consecutive items of one unit started
      bool ok = true, cont = false;
      int p = 0;
      Item item;
      // time accounting (trace builds): 2 waits for an image, 3 for a K tile and a free
      // logits buffer, 5 the whole loop, 6 tiles
      TRC_DECL(TR_CTA_SLOTS);
      TRC_T(tr_all);
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        if (!cont) {
          p = nrun & 1;
          TRC_T(tr_i);
          if (!mbar_wait(smem_u32(&imgready[p]), (nrun >> 1) & 1, ws, abort)) break;
          TRC_ADD(2, tr_i);
          tc_fence_after();
        }
        const uint64_t b0 = smem_desc_sw128(smem_u32(img + p * C::IMG_BYTES), 16, 1024);
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int st = it % KB_STAGES;
          const int ab = it % KB_NACC;
          TRC_T(tr_f);
          if (!mbar_wait(smem_u32(&full[kb_full<KB_STAGES>(it)]), kb_full_parity<KB_STAGES>(it), ws, abort) ||
              (it >= (uint32_t)KB_NACC &&
               !mbar_wait(smem_u32(&accempty[ab]), ((it / KB_NACC) & 1) ^ 1, ws, abort))) {
            ok = false;
            break;
          }
          TRC_ADD(3, tr_f);
          TRC_INC(6);
          tc_fence_after();
          // descriptors advance by (byte offset >> 4) in their address field
          const uint64_t a0 = smem_desc_sw128(smem_u32(tiles + st * KB_TILE_BYTES), 16, 1024);
          const uint32_t dl = tmem + ab * C::NB;
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {  // 16 channels per MMA
            const uint64_t ad = a0 + (uint64_t)((((k >> 2) * KB_BOX) + (k & 3) * 32) >> 4);
            const uint64_t bm = b0 + (uint64_t)((((k >> 2) * C::IMG_ATOM) + (k & 3) * 32) >> 4);
            umma_f16_ss(dl, ad, bm, C::IDESC, k > 0 ? 1u : 0u);
          }
          umma_commit(smem_u32(&empty[st]));
          umma_commit(smem_u32(&accfull[ab]));
        }
        if (!ok) break;
        cont = is.next_same_unit(item);
        if (!cont) {
          umma_commit(smem_u32(&imgfree[p]));
          ++nrun;
        }
      }
      // every MMA issued here completes before the CTA tears down tensor memory
      if (it > 0) mbar_wait(smem_u32(&accfull[(it - 1) % KB_NACC]), ((it - 1) / KB_NACC) & 1, ws, nullptr);
      TRC_ADD(5, tr_all);
      TRC_PUT(ws, TR_K_KPASS, 7);
    }
  } else if (warp == KB_BUILD_WARP) {
    // ------------------ mu' image and lambda, once per run, one run ahead
    uint32_t nrun = 0;
    bool cont = false;
    Item item;
    for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
      const bool same = cont;
      cont = is.next_same_unit(item);
      if (same) continue;  // the run's image is in place
      const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
      const int p = nrun & 1;
      if (nrun >= 2 && !mbar_wait(smem_u32(&imgfree[p]), ((nrun >> 1) - 1) & 1, ws, abort)) break;
      const int64_t qb = (((int64_t)item.seq * dm.L + l) * dm.Hq + (int64_t)g * G) * D;
      build_split_image<G>(img + p * C::IMG_BYTES, ws.mu + qb, lane);
      float* lam_s = lams + p * G * D;
      for (int e = lane; e < G * D / 4; e += 32) ((float4*)lam_s)[e] = ((const float4*)(ws.lam + qb))[e];
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&imgready[p]));
      ++nrun;
    }
  } else if (warp >= KB_KAPPA_WARP0 && warp < KB_READ_WARP0) {
    // ------------------------------------------------------ kappa ---------
    // A group's warp writes its partial kappa of all four token subsets into
    // the group's slot and signals kready; the readout warp of each subset
    // adds the four partials (in writer order) and stores the token's row.
    const int kw = warp - KB_KAPPA_WARP0;
    const int grp = kw >> 2;                  // tiles with it % 2 == grp
    const int cq = kw & 3;                    // channel quarter
    uint32_t it = 0, nrun = 0, ng = 0;        // ng: tiles of this group so far
    bool cont = false;
    int p = 0;
    Item item;
    // time accounting (trace builds, warp 2): 7 waits for a K tile, 8 its quarter
    // of kappa, 9 waits for the group's slot, 10 the partials into it, 11 the loop
    TRC_DECL(TR_CTA_SLOTS);
    TRC_T(tr_all);
    // Every wait is bounded and the warps meet at no named barrier, so a warp
    // whose wait failed (the abort flag is set) leaves on its own.
    for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
      if (!cont) {
        p = nrun & 1;
        if (!mbar_wait(smem_u32(&imgready[p]), (nrun >> 1) & 1, ws, abort)) goto kappa_done;
      }
      {
        const uint32_t lam_s = smem_u32(lams + p * G * D);
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          if ((int)(it & 1) != grp) continue;
          const int st = it % KB_STAGES;
          float part[4][G];
          TRC_T(tr_f);
          if (!mbar_wait(smem_u32(&full[kb_full<KB_STAGES>(it)]), kb_full_parity<KB_STAGES>(it), ws, abort))
            goto kappa_done;
          TRC_ADD(7, tr_f);
          TRC_T(tr_k);
          kappa_quarter<G>(smem_u32(tiles + st * KB_TILE_BYTES), lam_s, lane, cq, part);
          TRC_ADD(8, tr_k);
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&empty[st]));
          TRC_T(tr_b);
          // slot b of the group takes its tiles ng = b, b + SLOTS, ...; it is free
          // once the readout warps have read its previous tile
          const int b = ng % C::SLOTS, use = ng / C::SLOTS;
          const int ks = grp * C::SLOTS + b;
          if (use >= 1 && !mbar_wait(smem_u32(&kfree[ks]), (use - 1) & 1, ws, abort)) goto kappa_done;
          TRC_ADD(9, tr_b);
          TRC_T(tr_r);
          float* slot = kred + ks * C::SLOT_FLOATS;
#pragma unroll
          for (int j = 0; j < 4; ++j)
#pragma unroll
            for (int h = 0; h < G; ++h) slot[((j * 4 + cq) * G + h) * 32 + lane] = part[j][h];
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&kready[ks]));
          ++ng;
          TRC_ADD(10, tr_r);
        }
      }
      cont = is.next_same_unit(item);
      if (!cont) {
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&imgfree[p]));
        ++nrun;
      }
    }
  kappa_done:
    TRC_ADD(11, tr_all);
    if (warp == KB_KAPPA_WARP0 && lane == 0) TRC_PUT(ws, TR_K_KPASS, 12);
  } else if (warp >= KB_READ_WARP0 && warp < KB_READ_WARP0 + 4) {
    // ------------------------------------------ logits readout + stats ----
    const int quarter = warp & 3;
    const int y = quarter * 32 + lane;        // token row (tensor-memory lane)
    const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
    const int rw = warp - KB_READ_WARP0;
    uint32_t it = 0;
    bool bad = false, cont = false;
    float run_m[G], run_s[G];
    Item item;
    // time accounting (trace builds, first readout warp): 12 waits for logits, 13 the
    // readout of a tile (with 15, its wait for the kappa partials), 14 the whole loop
    TRC_DECL(TR_CTA_SLOTS);
    TRC_T(tr_all);
    for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
      if (!cont) {  // a new run of the unit's consecutive chunks: fresh statistics
#pragma unroll
        for (int h = 0; h < G; ++h) {
          run_m[h] = -INFINITY;
          run_s[h] = 0.f;
        }
      }
      float* lkp = ws.lk + (int64_t)item.plane * dm.Ntot * (2 * G);
      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        const int ab = it % KB_NACC;
        TRC_T(tr_f);
        if (!mbar_wait(smem_u32(&accfull[ab]), (it / KB_NACC) & 1, ws, abort)) break;  // abort: see below
        TRC_ADD(12, tr_f);
        TRC_T(tr_b);
        tc_fence_after();
        float dv[C::NB];
        if constexpr (C::NB == 16) tmem_ld16(tmem + ab * C::NB + lanes, dv);
        else tmem_ld32(tmem + ab * C::NB + lanes, dv);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&accempty[ab]));
        // kappa of this warp's 32 tokens: the four partials of the tile's group
        // (the group's slot holds [token subset][writer][G][32]), added in writer order
        const uint32_t ng = it >> 1;  // the tile is the ng-th of group it % 2
        const int ks = (int)(it & 1) * C::SLOTS + (int)(ng % C::SLOTS);
        TRC_T(tr_k);
        if (!mbar_wait(smem_u32(&kready[ks]), (ng / C::SLOTS) & 1, ws, abort)) break;  // abort: see below
        TRC_ADD(15, tr_k);
        const float* slot = kred + ks * C::SLOT_FLOATS;
        float row[2 * G];  // logits, then kappa
#pragma unroll
        for (int h = 0; h < G; ++h) {
          float v = 0.f;
#pragma unroll
          for (int q = 0; q < 4; ++q) v += slot[((quarter * 4 + q) * G + h) * 32 + lane];
          row[G + h] = v;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&kfree[ks]));
        const int64_t tok = t + y;
        if (tok < item.t1) {
#pragma unroll
          for (int h = 0; h < G; ++h) {
            const float lg = dv[h] + dv[G + h] + dv[2 * G + h];
            row[h] = lg;
            bad |= !isfinite(lg) || !isfinite(row[G + h]);
            // branch-free online update: one of the two exponentials is exp(0);
            // both arguments are <= 0, where the fast exponential's relative
            // error (a few ulp) is far below what the statistics need
            const float mn = fmaxf(run_m[h], lg);
            run_s[h] = run_s[h] * __expf(run_m[h] - mn) + __expf(lg - mn);
            run_m[h] = mn;
          }
          store_floats<2 * G, LkAlign<G>::ROW>(lkp + tok * (2 * G), row);
        }
        TRC_ADD(13, tr_b);
      }
      // ---- softmax statistics of a run, at its last chunk; the run's other
      // chunks get empty statistics (m = -inf, s = 0), which merge as nothing
      cont = is.next_same_unit(item);
      if (cont) {
        if (rw == 0 && lane < G) {
          float* cs = ws.cstats + (((int64_t)item.plane * dm.c_cap + item.cidx) * G + lane) * 2;
          cs[0] = -INFINITY;
          cs[1] = 0.f;
        }
        continue;
      }
#pragma unroll
      for (int h = 0; h < G; ++h) {
        softmax_warp_merge(run_m[h], run_s[h]);
        if (lane == 0) {
          red[rw * 2 * G + h] = run_m[h];
          red[rw * 2 * G + G + h] = run_s[h];
        }
      }
      // a warp that met an abort still arrives here; the barrier ORs the flag,
      // so all four leave together
      if (named_barrier_any(1, 128, *abort != 0)) goto read_done;
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
    TRC_ADD(14, tr_all);
    if (warp == KB_READ_WARP0 && lane == 0) TRC_PUT(ws, TR_K_KPASS, 16);
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
  JACAP_TRY(launch_pdl(dm.pdl != 0, kpass_bf16_kernel<G>, grid, KB_THREADS, smem, st, kmap, dm, ws, cu));
  return cudaGetLastError();
}

cudaError_t launch_kpass_bf16(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, const int32_t* cu, int grid,
                              cudaStream_t st) {
  switch (dm.G) {
    case 1: return launch_g<1>(kmap, dm, ws, cu, grid, st);
    case 2: return launch_g<2>(kmap, dm, ws, cu, grid, st);
    case 3: return launch_g<3>(kmap, dm, ws, cu, grid, st);
    case 4: return launch_g<4>(kmap, dm, ws, cu, grid, st);
    case 5: return launch_g<5>(kmap, dm, ws, cu, grid, st);
    case 6: return launch_g<6>(kmap, dm, ws, cu, grid, st);
    case 7: return launch_g<7>(kmap, dm, ws, cu, grid, st);
    case 8: return launch_g<8>(kmap, dm, ws, cu, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace jacap
