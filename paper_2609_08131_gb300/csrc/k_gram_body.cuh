// k_gram_body.cuh - the tcgen05 Gram pass as a device function: the
// kernel of k_gram.cu and the Gram role of the fused schedule (k_fused.cu)
// both run it. See k_gram.cu for what it computes.
#pragma once

#include "jacap_dev.cuh"

namespace jacap {


// Pool-softmax normaliser of the unit (plane, seq) for query head h of the
// group: M_h = max of the chunk maxima, Z_h = sum_c s_c exp(m_c - M_h). One
// warp: lanes take chunks c0 + lane + 32 k and a butterfly merges them in a
// fixed order, so the result does not depend on who computes it. The
// unit-statistics kernel runs it once per unit and head (ws.ustats).
template <int G>
__device__ __forceinline__ void unit_softmax_stats_warp(const Dims& dm, const Ws& ws, int plane, int seq, int h,
                                                        float& M, float& Z) {
  const int c0 = ws.plan[1 + seq], c1 = ws.plan[2 + seq];
  const float* cs = ws.cstats + ((int64_t)plane * dm.c_cap) * G * 2;
  float m = -INFINITY, s = 0.f;
  for (int c = c0 + (int)(threadIdx.x & 31); c < c1; c += 32)
    softmax_merge(m, s, cs[((int64_t)c * G + h) * 2], cs[((int64_t)c * G + h) * 2 + 1]);
  softmax_warp_merge(m, s);
  M = m;
  Z = s;
}

// The unit's (M_h, 1 / Z_h) of the G heads from ws.ustats into u[0 .. 2G):
// M_0 .. M_{G-1}, then 1/Z_0 .. 1/Z_{G-1}.
template <int G>
__device__ __forceinline__ void load_unit_stats(const Dims& dm, const Ws& ws, int plane, int seq, float (&u)[2 * G]) {
  const float* p = ws.ustats + ((int64_t)plane * dm.S + seq) * (2 * G);
#pragma unroll
  for (int e = 0; e < 2 * G; ++e) u[e] = p[e];
}

// --------------------------------------------------------------- tcgen05 ---
// G = sum_i v_i (w_i v_i)^T on the tensor cores with the scaled operand in
// tensor memory: D (128 x 128, fp32) += A (128 channels x 16 tokens, TMEM)
// * B (16 tokens x 128 channels, the TMA-staged V tile, MN-major). The TMA
// warp stages each V tile together with the tile's logits/kappa rows from the
// K pass (2G floats per token). The weight warp turns them into the Eq. 8
// weights (the same arithmetic as weight_kernel, with the unit's softmax
// statistics merged once per run), writes w for the score pass and leaves w
// as a bf16 pair hi + lo in the stage for the scaling warps. The scaling warps
// read V transposed with ldmatrix, form w_i v_i = hi + lo with packed bf16
// arithmetic and store hi and lo as two A operands; two MMAs per 16 tokens
// accumulate v hi^T and v lo^T, in two accumulators, each chain issued by a
// warp of its own: one thread's MMAs of N <= 128 follow each other at ~60 ns
// here whatever their accumulators, while two issuing threads overlap theirs.
// The epilogue adds the two.
// The scaling warps share nothing but the mbarriers of the pipeline. A run of
// consecutive chunks of one unit in a CTA's item range accumulates in the
// accumulator pair; four epilogue warps copy each finished run's Gram out
// before the next run starts on it.
constexpr int GR_THREADS = 544;   // warp 0: TMA, 1 and 16: MMA, 2-9: scale, 10-13: epilogue, 14-15: weights
constexpr int GR_MMA_LO_WARP = 16;  // issues the v lo^T chain (warp 1 the v hi^T chain)
constexpr int GR_EPI0 = 10;       // first epilogue warp
constexpr int GR_WEIGHT_WARP = 14;  // 14 and 15, 64 tokens of each tile each
constexpr int GR_SCALERS = 256;
constexpr int GR_BOX = 16384;      // {64 channels, 128 tokens} bf16, 128-byte swizzle
constexpr int GR_V_BYTES = 2 * GR_BOX;
constexpr int GR_W_BYTES = 512;    // the tile's weights as bf16 pairs, one word per token
constexpr uint32_t GR_TMEM_COLS = 512;
constexpr uint32_t GR_DLO = 128;   // accumulators: columns [0, 128) v hi^T, [128, 256) v lo^T
constexpr uint32_t GR_ACOL = 256;  // A buffers: [256 + 128 ab, +64) hi, [+64, +128) lo
// M = 128 (channels), N = 128 (channels), A in TMEM (K-major), B MN-major.
constexpr uint32_t GR_IDESC = idesc_bf16_f32(128, 128, 0, 1);

// RESERVE: shared memory the kernel needs besides the Gram's (the fused
// kernel's other roles' static variables), kept free when choosing stages.
template <int G, int RESERVE = 0>
struct GrCfg {
  static constexpr int LK_BYTES = TILE * 2 * G * 4 + 16;  // a tile's logits/kappa rows (+ alignment slack)
  static constexpr size_t smem_for(int stages) {
    return 1024 + (size_t)stages * (GR_V_BYTES + GR_W_BYTES + LK_BYTES) + 256;
  }
  static constexpr int VST = smem_for(6) + RESERVE <= 232448 ? 6 : 5;  // stages in flight
  static constexpr size_t SMEM = smem_for(VST);
  static_assert(SMEM + RESERVE <= 232448, "shared memory");
};

// The tile's logits/kappa rows (2G floats per token): the copy starts at the
// 16-byte boundary at or below the tile's first float (`off` floats before
// it) and covers the tile's `nvalid` tokens, rounded up to 16 bytes.
struct LkTile {
  int64_t f0;  // first copied float (multiple of 4)
  int off, nvalid;
  uint32_t bytes;
};
template <int G>
__device__ __forceinline__ LkTile lk_tile(const Dims& dm, const Item& item, int64_t t) {
  LkTile r;
  const int64_t a = ((int64_t)item.plane * dm.Ntot + t) * (2 * G);
  r.f0 = a & ~(int64_t)3;
  r.off = (int)(a - r.f0);
  r.nvalid = (int)(item.t1 - t < TILE ? item.t1 - t : TILE);
  r.bytes = (uint32_t)(((r.off + r.nvalid * 2 * G + 3) & ~3) * 4);
  return r;
}

// The Gram pass of CTA `part` of `parts` (all GR_THREADS threads of the CTA
// call it). FUSED: the role of the fused schedule (k_fused.cu): items strided
// over the role's CTAs, V tiles loaded with L2 policies (the first keep_tiles
// of an item evict_last, for the score role's second read, the rest and the
// rows evict_first), and every weight warp (per item) and epilogue warp (per
// run) adds its share to the unit's progress counter once its stores are
// visible device-wide: 6 per item in all.
template <int G, bool FUSED>
__device__ __forceinline__ void gram_bf16_body(const CUtensorMap* vmap_p, const Dims& dm, const Ws& ws, int part,
                                               int parts) {
  using C = GrCfg<G, FUSED ? 1024 : 0>;
  constexpr int GR_VST = C::VST;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* vring = smem;                                   // [GR_VST][GR_V_BYTES]
  uint8_t* wring = vring + GR_VST * GR_V_BYTES;            // [GR_VST][GR_W_BYTES] weight words
  uint8_t* lkring = wring + GR_VST * GR_W_BYTES;           // [GR_VST][LK_BYTES] logits/kappa rows
  uint64_t* vfull = (uint64_t*)(lkring + GR_VST * C::LK_BYTES);
  uint64_t* vempty = vfull + GR_VST;
  uint64_t* wready = vempty + GR_VST;  // the weight warp has written the tile's weights
  uint64_t* afull = wready + GR_VST;
  uint64_t* aempty = afull + 2;
  uint64_t* accfull = aempty + 2;   // the run's Gram is complete in the accumulators
  uint64_t* accempty = accfull + 1; // the epilogue has read them
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_skip;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_abort = 0;
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < GR_VST; ++i) {
      mbar_init(smem_u32(&vfull[i]), 1);
      mbar_init(smem_u32(&vempty[i]), 2);  // the two MMA warps' commits
      mbar_init(smem_u32(&wready[i]), 2);  // the two weight warps
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&afull[i]), GR_SCALERS / 32);
      mbar_init(smem_u32(&aempty[i]), 2);  // the two MMA warps' commits
    }
    mbar_init(smem_u32(accfull), 2);   // the two MMA warps' commits
    mbar_init(smem_u32(accempty), 4);  // the epilogue warps
    fence_mbar_init();
  }
  __syncthreads();
  if (s_skip) return;
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), GR_TMEM_COLS);
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
      prefetch_tmap(vmap_p);
      uint64_t keep = 0, drop = 0;
      const bool hints = FUSED && dm.keep_tiles >= 0;  // keep_tiles < 0: plain loads (tuning)
      if (hints) {
        keep = policy_evict_last();
        drop = policy_evict_first();
      }
      // time accounting (trace builds): 0 waits for a free stage, 1 the whole loop
      TRC_DECL(TR_CTA_SLOTS);
      TRC_T(tr_all);
      uint32_t it = 0;
      bool ok = true;
      Item item;
      for (ItemStream is(dm, ws, part, parts, FUSED); ok && is.next(item);) {
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        if (FUSED) JACAP_TRACE_MIN(ws, (int64_t)item.plane * dm.S + item.seq, TR_GRAM0);
        for (int64_t t = item.t0; t < item.t1; t += TILE) {
          const int st = it % GR_VST;
          TRC_T(tr_w);
          if (it >= (uint32_t)GR_VST &&
              !mbar_wait(smem_u32(&vempty[st]), ((it / GR_VST) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          TRC_ADD(0, tr_w);
          uint8_t* vt = vring + st * GR_V_BYTES;
          const LkTile lt = lk_tile<G>(dm, item, t);
          const uint32_t bar = smem_u32(&vfull[st]);
          mbar_arrive_expect_tx(bar, GR_V_BYTES + lt.bytes);
          if (hints) {
            const uint64_t pv = (t - item.t0) < (int64_t)dm.keep_tiles * TILE ? keep : drop;
            tma_load_4d_hint(smem_u32(vt), vmap_p, 0, (int)t, g, l, bar, pv);
            tma_load_4d_hint(smem_u32(vt + GR_BOX), vmap_p, 64, (int)t, g, l, bar, pv);
            bulk_g2s_hint(smem_u32(lkring + st * C::LK_BYTES), ws.lk + lt.f0, lt.bytes, bar, drop);
          } else {
            tma_load_4d(smem_u32(vt), vmap_p, 0, (int)t, g, l, bar);
            tma_load_4d(smem_u32(vt + GR_BOX), vmap_p, 64, (int)t, g, l, bar);
            bulk_g2s(smem_u32(lkring + st * C::LK_BYTES), ws.lk + lt.f0, lt.bytes, bar);
          }
          ++it;
        }
      }
      TRC_ADD(1, tr_all);
      TRC_PUT(ws, TR_K_GRAM, 2);
      for (uint32_t k = (it > (uint32_t)GR_VST ? it - GR_VST : 0); k < it; ++k)
        mbar_wait(smem_u32(&vfull[k % GR_VST]), (k / GR_VST) & 1, ws, nullptr);
    }
  } else if (warp == 1 || warp == GR_MMA_LO_WARP) {
    // ------------------------------------------------ MMA issuers ---------
    if (lane == 0) {
      const bool lo = warp == GR_MMA_LO_WARP;  // the v lo^T chain
      // time accounting (trace builds): 2 waits for a scaled operand, 3 for a free
      // accumulator (run start), 4 the whole loop, 5 tiles
      TRC_DECL(TR_CTA_SLOTS);
      TRC_T(tr_all);
      uint32_t it = 0, nrun = 0;
      bool ok = true, cont = false, first = true;
      Item item;
      for (ItemStream is(dm, ws, part, parts, FUSED); ok && is.next(item);) {
        // a run of consecutive chunks of a unit accumulates in the accumulator
        // pair; a new run starts on it once the previous run's epilogue has read it
        if (!cont) {
          TRC_T(tr_a);
          if (nrun >= 1 && !mbar_wait(smem_u32(accempty), (nrun - 1) & 1, ws, abort)) break;
          TRC_ADD(3, tr_a);
          tc_fence_after();
          first = true;
        }
        const uint32_t dacc = tmem + (lo ? GR_DLO : 0u);
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int vs = it % GR_VST, ab = it & 1;
          // the scaling warps arrive on afull only after the tile's V landed
          TRC_T(tr_f);
          if (!mbar_wait(smem_u32(&afull[ab]), (it >> 1) & 1, ws, abort)) {
            ok = false;
            break;
          }
          TRC_ADD(2, tr_f);
          TRC_INC(5);
          tc_fence_after();
          // B descriptors advance by (byte offset >> 4) in their address field
          const uint64_t b0 = smem_desc_sw128(smem_u32(vring + vs * GR_V_BYTES), GR_BOX, 1024);
          const uint32_t acol = tmem + GR_ACOL + 128 * ab + (lo ? 64u : 0u);  // hi or lo
#pragma unroll
          for (int k = 0; k < TILE / 16; ++k) {  // 16 tokens per MMA
            const uint64_t bd = b0 + (uint64_t)((k * 2048) >> 4);
            umma_f16_ts(dacc, acol + 8 * k, bd, GR_IDESC, (first && k == 0) ? 0u : 1u);
          }
          first = false;
          umma_commit(smem_u32(&vempty[vs]));
          umma_commit(smem_u32(&aempty[ab]));
        }
        if (!ok) break;
        cont = is.next_same_unit(item);
        if (!cont) {
          umma_commit(smem_u32(accfull));
          ++nrun;
        }
      }
      if (it > 0) mbar_wait(smem_u32(&aempty[(it - 1) & 1]), ((it - 1) >> 1) & 1, ws, nullptr);
      TRC_ADD(4, tr_all);
      if (!lo) TRC_PUT(ws, TR_K_GRAM, 6);
    }
  } else if (warp < 10) {
    // ------------------------------------------------- scaling warps ------
    const int quarter = warp & 3;        // TMEM lane quarter == channels 32 quarter .. +31
    const int th = (warp - 2) >> 2;      // token half of each tile (blocks 4 th .. 4 th + 3)
    // ldmatrix row addresses: lane l -> matrix l / 8, row l % 8
    const int lm = lane >> 3, lr = lane & 7;
    // time accounting (trace builds, warp 2): 6 waits for V, 7 for the weights,
    // 8 for a free operand buffer, 9 scaling, 10 the whole loop
    TRC_DECL(TR_CTA_SLOTS);
    TRC_T(tr_all);
    uint32_t it = 0;
    Item item;
    for (ItemStream is(dm, ws, part, parts, FUSED); is.next(item);) {
      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        const int vs = it % GR_VST, ab = it & 1;
        TRC_T(tr_v);
        if (!mbar_wait(smem_u32(&vfull[vs]), (it / GR_VST) & 1, ws, abort)) goto scale_done;
        TRC_ADD(6, tr_v);
        TRC_T(tr_wr);
        if (!mbar_wait(smem_u32(&wready[vs]), (it / GR_VST) & 1, ws, abort)) goto scale_done;
        TRC_ADD(7, tr_wr);
        // weights of this lane's token pairs (rows 2(l%4), 2(l%4)+1 of each
        // 8-token half of its 4 blocks) as bf16 pairs; tokens past the item
        // weigh zero
        uint32_t wph[8], wpl[8];
        {
          const int nvalid = (int)(item.t1 - t < TILE ? item.t1 - t : TILE);
          const uint32_t wsl = smem_u32(wring + vs * GR_W_BYTES);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int i0 = 16 * (4 * th + (e >> 1)) + 8 * (e & 1) + 2 * (lane & 3);
            const uint32_t x0 = i0 < nvalid ? lds_u32(wsl + 4 * i0) : 0u;
            const uint32_t x1 = i0 + 1 < nvalid ? lds_u32(wsl + 4 * i0 + 4) : 0u;
            wph[e] = __byte_perm(x0, x1, 0x5410);  // (hi of token i0, hi of i0 + 1)
            wpl[e] = __byte_perm(x0, x1, 0x7632);  // (lo, lo)
          }
        }
        TRC_T(tr_ae);
        if (it >= 2 && !mbar_wait(smem_u32(&aempty[ab]), ((it >> 1) & 1) ^ 1, ws, abort)) goto scale_done;
        TRC_ADD(8, tr_ae);
        TRC_T(tr_b);
        tc_fence_after();
        const uint32_t vt = smem_u32(vring + vs * GR_V_BYTES);
        const uint32_t acol = tmem + GR_ACOL + 128 * ab;
        // the tile's V fragments of this warp, all eight loads in flight
        // before any arithmetic or tensor-memory store (each store orders the
        // code around it); matrices: 0 = (tokens 0-7, ch c0..c0+7),
        // 1 = (tokens 0-7, c0+8..), 2 = (8-15, c0..), 3 = (8-15, c0+8..)
        uint32_t r[2][4][4];
#pragma unroll
        for (int lh = 0; lh < 2; ++lh)
#pragma unroll
          for (int blk = 0; blk < 4; ++blk) {
            const int b = 4 * th + blk;  // 16-token block of the tile
            const int c0 = quarter * 32 + lh * 16 + (lm & 1) * 8;
            const int tokr = 16 * b + (lm >> 1) * 8 + lr;
            const uint32_t addr = vt + (c0 >> 6) * GR_BOX + sw128_off(tokr, (c0 & 63) >> 3);
            ldsm_x4_trans(addr, r[lh][blk][0], r[lh][blk][1], r[lh][blk][2], r[lh][blk][3]);
          }
#pragma unroll
        for (int lh = 0; lh < 2; ++lh) {
          // one 32-column slab (this warp's 4 token blocks) of hi and of lo,
          // built in registers and written with one wide store each
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int blk = 0; blk < 4; ++blk)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              // w v = hi + lo; registers (r0 = lanes 0-7, r1 = lanes 8-15) of
              // columns 8 blk + 4 (q / 2) ..
              const int e = 4 * blk + 2 * (q >> 1) + (q & 1);
              bf16x2_scale_split(wph[2 * blk + (q >> 1)], wpl[2 * blk + (q >> 1)], r[lh][blk][q], hi[e], lo[e]);
            }
          const uint32_t lanes = (uint32_t)(quarter * 32 + lh * 16) << 16;
          tmem_st_16x128b_x8(acol + lanes + 32 * th, hi);
          tmem_st_16x128b_x8(acol + lanes + 64 + 32 * th, lo);
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&afull[ab]));
        TRC_ADD(9, tr_b);
      }
    }
  scale_done:;
    TRC_ADD(10, tr_all);
    if (warp == 2 && lane == 0) TRC_PUT(ws, TR_K_GRAM, 11);
  } else if (warp == GR_WEIGHT_WARP || warp == GR_WEIGHT_WARP + 1) {
    // ------------------------------------------------------ weights -------
    // Eq. 8 for the tile's tokens (two per lane of each of the two warps) from the staged logits and
    // kappa: w = wdiv sum_h rho_h^2 kappa_h, rho = alpha_bar (1 - alpha_bar),
    // alpha_bar = exp(l_h - M_h) / Z_h (rho = 1 for the linear surrogate);
    // (M_h, Z_h) merged from the unit's chunk statistics once per run.
    // time accounting (trace builds, first weight warp): 11 waits for V, 12 the
    // weights of a tile, 13 the whole loop
    TRC_DECL(TR_CTA_SLOTS);
    TRC_T(tr_all);
    uint32_t it = 0;
    bool bad = false, cont = false;
    float u[2 * G];  // M_h, then 1 / Z_h (from the unit-statistics kernel)
#pragma unroll
    for (int e = 0; e < 2 * G; ++e) u[e] = 0.f;
    Item item;
    for (ItemStream is(dm, ws, part, parts, FUSED); is.next(item);) {
      if (!cont && !dm.linear) load_unit_stats<G>(dm, ws, item.plane, item.seq, u);
      cont = is.next_same_unit(item);
      const int64_t base = (int64_t)item.plane * dm.Ntot;
      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        const int vs = it % GR_VST;
        TRC_T(tr_v);
        if (!mbar_wait(smem_u32(&vfull[vs]), (it / GR_VST) & 1, ws, abort)) goto weights_done;
        TRC_ADD(11, tr_v);
        TRC_T(tr_b);
        const LkTile lt = lk_tile<G>(dm, item, t);
        const float* rows = (const float*)(lkring + vs * C::LK_BYTES) + lt.off;
        uint32_t* wout = (uint32_t*)(wring + vs * GR_W_BYTES);
#pragma unroll
        for (int q = 0; q < 2; ++q) {
          const int i = 64 * (warp - GR_WEIGHT_WARP) + lane + 32 * q;
          uint32_t word = 0u;
          if (i < lt.nvalid) {
            float r[2 * G];
            // the staged copy keeps the rows' global alignment (off is the
            // row start's distance from the 16-byte boundary below it)
            load_floats<2 * G, LkAlign<G>::ROW>(r, rows + i * 2 * G);
            float wt = 0.f;
            if (dm.linear) {
#pragma unroll
              for (int h = 0; h < G; ++h) wt += r[G + h];
            } else {
#pragma unroll
              for (int h = 0; h < G; ++h) {
                const float a = expf(r[h] - u[h]) * u[G + h];  // alpha_bar
                const float rho = a * (1.f - a);                // diagonal of the softmax Jacobian
                wt = fmaf(rho * rho, r[G + h], wt);             // rho^2 kappa
              }
            }
            wt *= dm.wdiv;
            bad |= !isfinite(wt);
            ws.w[base + t + i] = wt;
            // hi = RN(w), lo = RN(w - hi) (w - hi is exact in float32)
            word = pack_bf16x2(wt, wt - bf16lo(pack_bf16x2(wt, 0.f)));
          }
          wout[i] = word;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&wready[vs]));
        TRC_ADD(12, tr_b);
      }
      if (FUSED) {  // this warp's weights of the item are stored: its share of the unit's progress
        __threadfence();
        __syncwarp();
        if (lane == 0) red_add_release_gpu(ws.gcount + (int64_t)item.plane * dm.S + item.seq, 1);
      }
    }
  weights_done:
    TRC_ADD(13, tr_all);
    if (warp == GR_WEIGHT_WARP && lane == 0) TRC_PUT(ws, TR_K_GRAM, 14);
    if (bad) flag(ws, ST_NONFINITE);
  } else {
    // ------------------------------------------------------ epilogue ------
    // The accumulator pair holds a run's partial Gram (v hi^T + v lo^T); warp
    // (quarter q) copies rows 32 q .. +31, each lane its row: 32 consecutive
    // floats per column block, so a lane writes 128 contiguous bytes per
    // block. The Gram is symmetric and its consumers read the lower triangle
    // only, so only the column blocks cb <= q (the lower 32 x 32 blocks) are
    // written.
    const int quarter = warp & 3;
    const int m = quarter * 32 + lane;
    uint32_t nrun = 0;
    bool cont = false;
    int run_cidx = 0, run_items = 0;
    Item item;
    for (ItemStream is(dm, ws, part, parts, FUSED); is.next(item);) {
      // the partial of a run goes to its first chunk; pflag marks which
      // chunks hold one
      if (!cont) {
        run_cidx = item.cidx;
        run_items = 0;
      }
      ++run_items;
      if (warp == GR_EPI0 && lane == 0) ws.pflag[(int64_t)item.plane * dm.c_cap + item.cidx] = cont ? 0 : 1;
      cont = is.next_same_unit(item);
      if (cont) continue;
      if (!mbar_wait(smem_u32(accfull), nrun & 1, ws, abort)) break;
      tc_fence_after();
      const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
      float* dst = ws.gpart + ((int64_t)item.plane * dm.c_cap + run_cidx) * D * D + (int64_t)m * 32;
#pragma unroll 1
      for (int cb = 0; cb <= quarter; ++cb) {
        float a[32], b[32];
        tmem_ld32(trow + cb * 32, a);
        tmem_ld32(trow + GR_DLO + cb * 32, b);
#pragma unroll
        for (int j = 0; j < 32; j += 4)
          *(float4*)(dst + cb * D * 32 + j) =
              make_float4(a[j] + b[j], a[j + 1] + b[j + 1], a[j + 2] + b[j + 2], a[j + 3] + b[j + 3]);
      }
      tc_fence_before();
      if (FUSED) __threadfence();  // this warp's rows of the partial (and the pflag entries) are visible
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(accempty));
      if (FUSED && lane == 0) {
        red_add_release_gpu(ws.gcount + (int64_t)item.plane * dm.S + item.seq, run_items);
        JACAP_TRACE_MAX(ws, (int64_t)item.plane * dm.S + item.seq, TR_GRAM1);
      }
      ++nrun;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, GR_TMEM_COLS);
  }
}

}  // namespace jacap
