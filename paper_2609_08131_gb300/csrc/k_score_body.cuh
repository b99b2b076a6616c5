// k_score_body.cuh - the tcgen05 score pass as a device function: the
// kernel of k_score.cu and the score role of the fused schedule (k_fused.cu)
// both run it. See k_score.cu for what it computes.
#pragma once

#include "jacap_dev.cuh"

namespace jacap {


// warp 0: V tiles (TMA), 1: MMA, 2-5 and 7-10: epilogue (two warps per tensor-memory
// lane quarter, each half of the accumulator's columns), 6: images
constexpr int SC_THREADS = 352;
constexpr int SC_EPI_B0 = 7;  // first warp of the second epilogue group
template <bool DENSE> __host__ __device__ constexpr int sc_stages() { return DENSE ? 3 : 4; }  // V tiles in flight
template <bool DENSE> __host__ __device__ constexpr int sc_imgs() { return 2; }  // L^{-1} image buffers
constexpr int SC_BOX = 16384;
constexpr int SC_TILE_BYTES = 2 * SC_BOX;
constexpr int SC_M_BYTES = 65536;
// Accumulators: DENSE, two of 128 columns (hi and lo of the matrix add into
// one); lower-triangular L^{-1}, two of 256 columns (hi and lo of each output
// row in separate columns, see below).
template <bool DENSE> __host__ __device__ constexpr uint32_t sc_tmem_cols() { return DENSE ? 256 : 512; }
template <bool DENSE> __host__ __device__ constexpr uint32_t sc_acc_cols() { return DENSE ? 128 : 256; }
// DENSE: M = 128 tokens, N = 128 rows of the image, both operands K-major.
constexpr uint32_t SC_IDESC128 = idesc_bf16_f32(128, 128, 0, 0);
// Lower-triangular L^{-1}: the image interleaves hi and lo by 16-row blocks
// (image row 32 b + 16 p + t holds part p of output row 16 b + t), so the
// K-step of channels 16 k .. 16 k + 15, which feeds only output rows >= 16 k,
// is one MMA over image rows 32 k .. 255: N = 256 - 32 k, accumulator columns
// 32 k .. 255 (620 tensor cycles per tile against 880 for hi and lo in
// separate MMAs with the triangle cut at 64 rows).
__host__ __device__ constexpr uint32_t sc_idesc_tri(int k) { return idesc_bf16_f32(128, 256 - 32 * k, 0, 0); }

// the lower-triangular image in shared memory: channel atom 0 whole (32 KB),
// then rows 128-255 of atom 1 (16 KB; its rows 0-127 belong to output rows
// 0-63, which have no channel >= 64)
constexpr int SC_MT_BYTES = 49152;
template <bool DENSE> __host__ __device__ constexpr int sc_img_bytes() { return DENSE ? SC_M_BYTES : SC_MT_BYTES; }
template <bool DENSE>
constexpr size_t score_bf16_smem_bytes() {
  // + 17 mbarriers (136 B, rounded to 144) + the epilogue groups' partial sums (2 x 128 floats)
  return 1024 + sc_imgs<DENSE>() * sc_img_bytes<DENSE>() + sc_stages<DENSE>() * SC_TILE_BYTES + 144 + 1024;
}

// DENSE: the score matrix is a full 128 x 128 (output directions) rather than
// the lower-triangular L^{-1}, so no K-step may be narrowed.
// The score pass of CTA `part` of `parts` (warps 0-10 work; further warps of
// the CTA only meet its barriers). FUSED: the role of the fused schedule
// (k_fused.cu): items strided over the role's CTAs, V tiles loaded with the L2
// evict_first policy (the Gram role left the first tiles of each item in L2),
// and a unit's image and weights are read only once the factor role has
// published the unit (fdone).
template <bool DENSE, bool FUSED>
__device__ __forceinline__ void score_bf16_body(const CUtensorMap* vmap_p, const Dims& dm, const Ws& ws,
                                                float* __restrict__ scores, int part, int parts) {
  constexpr int SC_STAGES = sc_stages<DENSE>();
  constexpr int SC_IMGS = sc_imgs<DENSE>();
  constexpr int IMG = sc_img_bytes<DENSE>();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* mimg = smem;                       // [SC_IMGS][IMG], by run
  uint8_t* stages = smem + SC_IMGS * IMG;
  uint64_t* vfull = (uint64_t*)(stages + SC_STAGES * SC_TILE_BYTES);
  uint64_t* vempty = vfull + SC_STAGES;
  uint64_t* accfull = vempty + SC_STAGES;
  uint64_t* accempty = accfull + 2;
  uint64_t* mfull = accempty + 2;   // [2]
  uint64_t* mempty = mfull + 2;     // [2]
  uint64_t* mdone = mempty + 2;
  float* s_part = (float*)(stages + SC_STAGES * SC_TILE_BYTES + 144);  // [2][128] second group's partial sums
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_skip;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_abort = 0;
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < SC_STAGES; ++i) {
      mbar_init(smem_u32(&vfull[i]), 1);
      mbar_init(smem_u32(&vempty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&accfull[i]), 1);
      mbar_init(smem_u32(&accempty[i]), 8);  // the eight epilogue warps
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&mfull[i]), 1);
      mbar_init(smem_u32(&mempty[i]), 1);
    }
    mbar_init(smem_u32(mdone), 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (s_skip) return;
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), sc_tmem_cols<DENSE>());
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  volatile int* abort = &s_abort;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(vmap_p);
      const bool hints = FUSED && dm.keep_tiles >= 0;  // keep_tiles < 0: plain loads (tuning)
      const uint64_t drop = hints ? policy_evict_first() : 0;
      uint32_t it = 0;
      bool ok = true;
      Item item;
      // time accounting (trace builds): 0 waits for a free stage, 1 the whole loop
      TRC_DECL(TR_CTA_SLOTS);
      TRC_T(tr_all);
      for (ItemStream is(dm, ws, part, parts, FUSED); ok && is.next(item);) {
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        for (int64_t t = item.t0; t < item.t1; t += TILE) {
          const int st = it % SC_STAGES;
          TRC_T(tr_w);
          if (it >= (uint32_t)SC_STAGES &&
              !mbar_wait(smem_u32(&vempty[st]), ((it / SC_STAGES) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          TRC_ADD(0, tr_w);
          uint8_t* vt = stages + st * SC_TILE_BYTES;
          mbar_arrive_expect_tx(smem_u32(&vfull[st]), SC_TILE_BYTES);
          if (hints) {
            tma_load_4d_hint(smem_u32(vt), vmap_p, 0, (int)t, g, l, smem_u32(&vfull[st]), drop);
            tma_load_4d_hint(smem_u32(vt + SC_BOX), vmap_p, 64, (int)t, g, l, smem_u32(&vfull[st]), drop);
          } else {
            tma_load_4d(smem_u32(vt), vmap_p, 0, (int)t, g, l, smem_u32(&vfull[st]));
            tma_load_4d(smem_u32(vt + SC_BOX), vmap_p, 64, (int)t, g, l, smem_u32(&vfull[st]));
          }
          ++it;
        }
      }
      TRC_ADD(1, tr_all);
      TRC_PUT(ws, TR_K_SCORE, 2);
      for (uint32_t k = (it > (uint32_t)SC_STAGES ? it - SC_STAGES : 0); k < it; ++k)
        mbar_wait(smem_u32(&vfull[k % SC_STAGES]), (k / SC_STAGES) & 1, ws, nullptr);
    }
  } else if (warp == 6) {
    // ------------------- the L^{-1} image of each run, into the buffer of the run SC_IMGS runs back
    // (a warp of its own, so the V tiles never wait behind an image slot)
    if (lane == 0) {
      uint32_t nrun = 0;
      bool cont = false;
      Item item;
      for (ItemStream is(dm, ws, part, parts, FUSED); is.next(item);) {
        const bool same = cont;
        cont = is.next_same_unit(item);
        if (same) continue;
        const int64_t u = (int64_t)item.plane * dm.S + item.seq;
        const int mp = nrun % SC_IMGS;
        if (nrun >= SC_IMGS && !mbar_wait(smem_u32(&mempty[mp]), ((nrun / SC_IMGS) & 1) ^ 1, ws, abort)) break;
        if (FUSED) {  // the factor role has published the unit's image
          if (!wait_count(ws.fdone + u, 1, ws, abort)) break;
          fence_proxy_async_global();
          JACAP_TRACE_MIN(ws, u, TR_SC_IMG);
        }
        mbar_arrive_expect_tx(smem_u32(&mfull[mp]), IMG);
        const uint8_t* src = ws.minv_img + u * SC_M_BYTES;
        uint8_t* dst = mimg + mp * IMG;
        if (DENSE) {
          bulk_g2s(smem_u32(dst), src, SC_M_BYTES, smem_u32(&mfull[mp]));
        } else {
          bulk_g2s(smem_u32(dst), src, 32768, smem_u32(&mfull[mp]));
          bulk_g2s(smem_u32(dst + 32768), src + 32768 + 16384, 16384, smem_u32(&mfull[mp]));
        }
        ++nrun;
      }
      for (uint32_t k = (nrun > (uint32_t)SC_IMGS ? nrun - SC_IMGS : 0); k < nrun; ++k)
        mbar_wait(smem_u32(&mfull[k % SC_IMGS]), (k / SC_IMGS) & 1, ws, nullptr);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      uint32_t it = 0, nrun = 0;
      bool ok = true, cont = false;
      int mp = 0;
      Item item;
      // time accounting (trace builds): 2 waits for an image, 3 for a free
      // accumulator, 4 for a V tile, 5 the whole loop, 6 tiles
      TRC_DECL(TR_CTA_SLOTS);
      TRC_T(tr_all);
      for (ItemStream is(dm, ws, part, parts, FUSED); ok && is.next(item);) {
        if (!cont) {
          mp = nrun % SC_IMGS;
          TRC_T(tr_m);
          if (!mbar_wait(smem_u32(&mfull[mp]), (nrun / SC_IMGS) & 1, ws, abort)) break;
          TRC_ADD(2, tr_m);
          tc_fence_after();
          if (FUSED) JACAP_TRACE_MIN(ws, (int64_t)item.plane * dm.S + item.seq, TR_SC_MMA);
        }
        const uint32_t ma = smem_u32(mimg + mp * IMG);
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int st = it % SC_STAGES;
          const int ab = it & 1;
          TRC_T(tr_a);
          if (it >= 2 && !mbar_wait(smem_u32(&accempty[ab]), ((it >> 1) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          TRC_ADD(3, tr_a);
          TRC_T(tr_v);
          if (!mbar_wait(smem_u32(&vfull[st]), (it / SC_STAGES) & 1, ws, abort)) {
            ok = false;
            break;
          }
          TRC_ADD(4, tr_v);
          TRC_INC(6);
          tc_fence_after();
          // descriptors advance by (byte offset >> 4); image rows: hi at row n,
          // lo at row 128 + n (16 KB further) of each 32 KB channel atom
          const uint64_t a0 = smem_desc_sw128(smem_u32(stages + st * SC_TILE_BYTES), 16, 1024);
          const uint64_t b0 = smem_desc_sw128(ma, 16, 1024);
          const uint32_t dacc = tmem + ab * sc_acc_cols<DENSE>();
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {  // 16 channels per K-step
            const uint64_t ad = a0 + (uint64_t)((((k >> 2) * SC_BOX) + (k & 3) * 32) >> 4);
            if (DENSE) {  // a full matrix: hi (rows 0-127) and lo (rows 128-255) into the same 128 columns
              const uint64_t bk = b0 + (uint64_t)((((k >> 2) * 32768) + (k & 3) * 32) >> 4);
              umma_f16_ss(dacc, ad, bk, SC_IDESC128, k > 0 ? 1u : 0u);
              umma_f16_ss(dacc, ad, bk + (16384 >> 4), SC_IDESC128, 1u);
            } else {  // image rows 32 k .. 255 (atom 1 is stored from its row 128)
              const uint64_t bk = b0 + (uint64_t)(((k < 4 ? 4096 * k : 32768 + 4096 * (k - 4)) + (k & 3) * 32) >> 4);
              umma_f16_ss(dacc + 32 * k, ad, bk, sc_idesc_tri(k), k > 0 ? 1u : 0u);
            }
          }
          umma_commit(smem_u32(&vempty[st]));
          umma_commit(smem_u32(&accfull[ab]));
        }
        if (!ok) break;
        cont = is.next_same_unit(item);
        if (!cont) {  // the run's last MMAs read the image: release it after them
          umma_commit(smem_u32(&mempty[mp]));
          ++nrun;
        }
      }
      // every MMA issued by this thread has completed before teardown
      umma_commit(smem_u32(mdone));
      mbar_wait(smem_u32(mdone), 0, ws, nullptr);
      TRC_ADD(5, tr_all);
      TRC_PUT(ws, TR_K_SCORE, 7);
    }
  } else if (warp < 6 || (warp >= SC_EPI_B0 && warp < SC_EPI_B0 + 4)) {
    // Epilogue: warp w reads tensor-memory lanes 32 (w % 4) .. + 31 (one token
    // per thread). Group 0 (warps 2-5) reduces the first half of the
    // accumulator's columns, group 1 (warps 7-10) the second half and leaves
    // its partial sums in shared memory; the two warps of a lane quarter meet
    // at a named barrier (1 + quarter) per tile and group 0 adds, multiplies
    // by w and stores the score. A warp whose wait failed still meets its
    // partner at the tile's barrier; both leave after it.
    const int quarter = warp & 3;
    const int grp = warp < 6 ? 0 : 1;
    const int y = quarter * 32 + lane;  // token row of the tile == TMEM lane
    constexpr int HALF = sc_acc_cols<DENSE>() / 2;
    uint32_t it = 0;
    bool bad = false, cont = false;
    Item item;
    // time accounting (trace builds, warp 2): 7 waits for an accumulator,
    // 8 reading and reducing it, 9 the rest of the tile, 10 the whole loop
    TRC_DECL(TR_CTA_SLOTS);
    TRC_T(tr_all);
    for (ItemStream is(dm, ws, part, parts, FUSED); is.next(item);) {
      bool unit_ok = true;
      if (FUSED && !cont && grp == 0) {  // the unit's weights are complete once its factor is published
        if (lane == 0) unit_ok = wait_count(ws.fdone + (int64_t)item.plane * dm.S + item.seq, 1, ws, abort);
        unit_ok = __shfl_sync(0xffffffffu, unit_ok ? 1 : 0, 0) != 0;
        if (!unit_ok && lane == 0) *abort = 1;  // the partner leaves after the next barrier
        __syncwarp();  // the lanes' loads of w come after lane 0's acquire
      }
      cont = is.next_same_unit(item);
      // group 0 loads each tile's w two tiles ahead, into two registers used in
      // turn (the loop takes two tiles per round), so the loads' latency, about
      // a tile's time, overlaps the reductions of the tiles before them
      const float* wrow = ws.w + (int64_t)item.plane * dm.Ntot + y;
      auto wload = [&](int64_t tt) -> float { return (grp == 0 && unit_ok && tt + y < item.t1) ? wrow[tt] : 0.f; };
      // one tile; false once the epilogue has to stop
      auto tile = [&](int64_t t, float wt) -> bool {
        const int ab = it & 1;
        const int64_t tok = t + y;
        TRC_T(tr_f);
        const bool ok = unit_ok && mbar_wait(smem_u32(&accfull[ab]), (it >> 1) & 1, ws, abort);
        TRC_ADD(7, tr_f);
        TRC_T(tr_r);
        float ssq = 0.f;
        if (ok) {
          tc_fence_after();
          const uint32_t trow =
              tmem + ab * sc_acc_cols<DENSE>() + grp * HALF + ((uint32_t)(quarter * 32) << 16);
          if (DENSE) {
#pragma unroll 1
            for (int cb = 0; cb < HALF / 32; ++cb) {
              float a[32];
              tmem_ld32(trow + cb * 32, a);
#pragma unroll
              for (int j = 0; j < 32; ++j) ssq = fmaf(a[j], a[j], ssq);
            }
          } else {  // y = hi + lo, block by block: columns 32 b + t and 32 b + 16 + t
#pragma unroll 1
            for (int cb = 0; cb < HALF / 32; cb += 2) {
              uint32_t a[32], b2[32];
              tmem_ld32x2(trow + cb * 32, trow + cb * 32 + 32, a, b2);
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                const float y0 = __uint_as_float(a[j]) + __uint_as_float(a[16 + j]);
                const float y1 = __uint_as_float(b2[j]) + __uint_as_float(b2[16 + j]);
                ssq = fmaf(y0, y0, ssq);
                ssq = fmaf(y1, y1, ssq);
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&accempty[ab]));
          if (grp == 1) s_part[ab * TILE + y] = ssq;
        }
        // the pair decides together whether to leave (see named_barrier_any)
        const bool stop = named_barrier_any(1 + quarter, 64, !ok || *abort != 0);
        TRC_ADD(8, tr_r);
        if (stop) return false;
        TRC_T(tr_s);
        if (grp == 0 && tok < item.t1) {
          const float sc = wt * (ssq + s_part[ab * TILE + y]);
          scores[(int64_t)item.plane * dm.Ntot + tok] = sc;
          bad |= !isfinite(sc);
        }
        TRC_ADD(9, tr_s);
        ++it;
        return true;
      };
      float w0 = wload(item.t0), w1 = wload(item.t0 + TILE);
      bool go = true;
      for (int64_t t = item.t0; go && t < item.t1; t += 2 * TILE) {
        go = tile(t, w0);
        w0 = wload(t + 2 * TILE);
        if (go && t + TILE < item.t1) {
          go = tile(t + TILE, w1);
          w1 = wload(t + 3 * TILE);
        }
      }
      if (!go) goto epi_done;
      if (FUSED && grp == 0 && lane == 0) JACAP_TRACE_MAX(ws, (int64_t)item.plane * dm.S + item.seq, TR_SC1);
    }
  epi_done:
    TRC_ADD(10, tr_all);
    if (warp == 2 && lane == 0) TRC_PUT(ws, TR_K_SCORE, 11);
    if (bad) flag(ws, ST_NONFINITE);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, sc_tmem_cols<DENSE>());
  }
}

}  // namespace jacap
