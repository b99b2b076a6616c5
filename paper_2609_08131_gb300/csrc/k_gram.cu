// k_gram.cu - fused Jacobian weight + weighted Gram pass over V.
//
// For every work item (a chunk of one unit's tokens) this pass
//   1. combines the K pass's per-chunk (max, sum exp) into the pool-softmax
//      normaliser (M_h, Z_h) of each query head h of the group (Sec. 3.4,
//      display after Algorithm 1);
//   2. forms w_i = (1/d) sum_h [alpha_bar (1 - alpha_bar)]^2 kappa_h,i with
//      alpha_bar = exp(l_h,i - M_h) / Z_h (Eq. 8; GQA heads summed) and stores
//      w for the score pass;
//   3. accumulates the chunk's partial Gram  sum_i w_i v_i v_i^T  (Eq. 9).
//
// bf16 caches use the 5th-generation tensor cores. B = V straight from the
// TMA-staged tile (bf16 is exact); the scaled operand w_i v_i = hi + lo is
// split into two bf16 halves (residual ~2^-17 relative per product) by the
// scaling warps and written to tensor memory as two A operands, so
// D = sum_i (hi_i + lo_i) v_i^T accumulates in fp32 in tensor memory without
// passing the scaled operand through shared memory. float32 caches take a
// SIMT fp32 kernel of the same contract.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

// Pool-softmax normaliser of the unit (plane, seq) for G heads: M_h = max of the
// chunk maxima, Z_h = sum_c s_c exp(m_c - M_h), combined in chunk order.
// Same normaliser computed by one warp: lanes take chunks c0 + lane + 32 k and
// a butterfly merges them (fixed order, so every CTA of the unit agrees).
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

template <int G>
__device__ __forceinline__ void unit_softmax_stats(const Dims& dm, const Ws& ws, int plane, int seq, int h,
                                                   float& M, float& Z) {
  const int c0 = ws.plan[1 + seq], c1 = ws.plan[2 + seq];
  const float* cs = ws.cstats + ((int64_t)plane * dm.c_cap) * G * 2;
  M = -INFINITY;
  for (int c = c0; c < c1; ++c) M = fmaxf(M, cs[((int64_t)c * G + h) * 2]);
  Z = 0.f;
  for (int c = c0; c < c1; ++c) {
    const float m = cs[((int64_t)c * G + h) * 2];
    if (m > -INFINITY) Z += cs[((int64_t)c * G + h) * 2 + 1] * expf(m - M);
  }
}

// w_i of Eq. 8 summed over the G query heads of the group (reading: GQA heads
// add their weights). ustat = [M_0..M_{G-1}, Z_0..Z_{G-1}].
template <int G>
__device__ __forceinline__ void load_lk(const Dims& dm, const Ws& ws, int plane, int64_t tok, float* lk) {
  const float* src = ws.lk + ((int64_t)plane * dm.Ntot + tok) * (2 * G);
  if constexpr ((2 * G) % 4 == 0) {
#pragma unroll
    for (int e = 0; e < 2 * G; e += 4) {
      const float4 q4 = *(const float4*)(src + e);
      lk[e] = q4.x; lk[e + 1] = q4.y; lk[e + 2] = q4.z; lk[e + 3] = q4.w;
    }
  } else {
#pragma unroll
    for (int e = 0; e < 2 * G; ++e) lk[e] = src[e];
  }
}

template <int G>
__device__ __forceinline__ float weight_from_lk(const Dims& dm, const float* ustat, const float* lk) {
  float wt = 0.f;
#pragma unroll
  for (int h = 0; h < G; ++h) {
    const float a = expf(lk[h] - ustat[h]) / ustat[G + h];  // alpha_bar
    const float rho = a * (1.f - a);                           // diagonal of S
    wt = fmaf(rho * rho, lk[G + h], wt);                       // rho^2 kappa
  }
  return wt * dm.wdiv;
}

// Logits and kappa of heads h0 .. h0 + NH - 1 of one token (src points at
// the token's row + h0).
template <int G, int NH>
__device__ __forceinline__ void load_lk_part(const float* src, float (&l)[NH], float (&k)[NH]) {
#pragma unroll
  for (int j = 0; j < NH; ++j) {
    l[j] = src[j];
    k[j] = src[G + j];
  }
}

// Partial Eq. 8 sum over heads h0 .. h0 + NH - 1 from the logits/kappa row;
// uinv = [M_0..M_{G-1}, 1/Z_0..1/Z_{G-1}] (the reciprocal saves a divide per head).
template <int G, int NH>
__device__ __forceinline__ float weight_part(const float* l, const float* kap, const float* uinv, int h0) {
  float wt = 0.f;
#pragma unroll
  for (int j = 0; j < NH; ++j) {
    const float a = expf(l[j] - uinv[h0 + j]) * uinv[G + h0 + j];  // alpha_bar
    const float rho = a * (1.f - a);                                  // diagonal of S
    wt = fmaf(rho * rho, kap[j], wt);                                 // rho^2 kappa
  }
  return wt;
}

template <int G>
__device__ __forceinline__ float jacobian_weight(const Dims& dm, const Ws& ws, const float* ustat, int plane,
                                                 int64_t tok) {
  float lk[2 * G];
  load_lk<G>(dm, ws, plane, tok, lk);
  return weight_from_lk<G>(dm, ustat, lk);
}

// --------------------------------------------------------------- tcgen05 ---
// G = sum_i v_i (w_i v_i)^T on the tensor cores with the scaled operand in
// tensor memory: D (128 x 128, fp32) += A (128 channels x 16 tokens, TMEM)
// * B (16 tokens x 128 channels, the TMA-staged V tile, MN-major). Per tile
// the scaling warps read V transposed with ldmatrix, multiply by w_i, split
// w_i v_i = hi + lo (bf16 each) and store hi and lo as two A operands; two
// MMAs per 16 tokens accumulate v (hi + lo)^T.
constexpr int GR_THREADS = 320;   // warp 0: TMA, warp 1: MMA, warps 2-9: scale + epilogue
constexpr int GR_SCALERS = 256;
constexpr int GR_VST = 6;          // V tiles in flight
constexpr int GR_BOX = 16384;      // {64 channels, 128 tokens} bf16, 128-byte swizzle
constexpr int GR_V_BYTES = 2 * GR_BOX;
constexpr uint32_t GR_TMEM_COLS = 512;
constexpr uint32_t GR_ACOL = 128;  // A buffers: [128 + 128 ab, +64) hi, [+64, +128) lo
// M = 128 (channels), N = 128 (channels), A in TMEM (K-major), B MN-major.
constexpr uint32_t GR_IDESC = idesc_bf16_f32(128, 128, 0, 1);

constexpr size_t gram_bf16_smem_bytes() { return 1024 + GR_VST * GR_V_BYTES + GR_VST * TILE * 4 + 256; }

template <int G>
__global__ void __launch_bounds__(GR_THREADS, 1)
    gram_bf16_kernel(const __grid_constant__ CUtensorMap vmap, Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* vring = smem;                                        // [GR_VST][GR_V_BYTES]
  float* wbuf = (float*)(vring + GR_VST * GR_V_BYTES);          // [GR_VST][TILE] weights of the tile
  float* ustat = wbuf + GR_VST * TILE;                          // [2G] (<= 16 floats)
  uint64_t* vfull = (uint64_t*)(ustat + 16);
  uint64_t* vempty = vfull + GR_VST;
  uint64_t* afull = vempty + GR_VST;
  uint64_t* aempty = afull + 2;
  uint64_t* accfull = aempty + 2;
  uint64_t* accempty = accfull + 1;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_skip;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_abort = 0;
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < GR_VST; ++i) {
      mbar_init(smem_u32(&vfull[i]), 1);
      mbar_init(smem_u32(&vempty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&afull[i]), GR_SCALERS / 32);
      mbar_init(smem_u32(&aempty[i]), 1);
    }
    mbar_init(smem_u32(accfull), 1);
    mbar_init(smem_u32(accempty), GR_SCALERS / 32);
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
      prefetch_tmap(&vmap);
      uint32_t it = 0;
      bool ok = true;
      Item item;
      for (int64_t i = blockIdx.x; ok && decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        for (int64_t t = item.t0; t < item.t1; t += TILE) {
          const int st = it % GR_VST;
          if (it >= (uint32_t)GR_VST &&
              !mbar_wait(smem_u32(&vempty[st]), ((it / GR_VST) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          uint8_t* vt = vring + st * GR_V_BYTES;
          mbar_arrive_expect_tx(smem_u32(&vfull[st]), GR_V_BYTES);
          tma_load_4d(smem_u32(vt), &vmap, 0, (int)t, g, l, smem_u32(&vfull[st]));
          tma_load_4d(smem_u32(vt + GR_BOX), &vmap, 64, (int)t, g, l, smem_u32(&vfull[st]));
          ++it;
        }
      }
      for (uint32_t k = (it > (uint32_t)GR_VST ? it - GR_VST : 0); k < it; ++k)
        mbar_wait(smem_u32(&vfull[k % GR_VST]), (k / GR_VST) & 1, ws, nullptr);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer ----------
    if (lane == 0) {
      uint32_t it = 0, nitem = 0;
      bool ok = true;
      Item item;
      for (int64_t i = blockIdx.x; ok && decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
        if (nitem > 0 && !mbar_wait(smem_u32(accempty), (nitem - 1) & 1, ws, abort)) break;
        tc_fence_after();
        bool first = true;
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int vs = it % GR_VST, ab = it & 1;
          if (!mbar_wait(smem_u32(&vfull[vs]), (it / GR_VST) & 1, ws, abort) ||
              !mbar_wait(smem_u32(&afull[ab]), (it >> 1) & 1, ws, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t va = smem_u32(vring + vs * GR_V_BYTES);
          const uint32_t acol = tmem + GR_ACOL + 128 * ab;
#pragma unroll
          for (int k = 0; k < TILE / 16; ++k) {  // 16 tokens per MMA
            const uint64_t bd = smem_desc_sw128(va + k * 2048, GR_BOX, 1024);
            umma_f16_ts(tmem, acol + 8 * k, bd, GR_IDESC, (first && k == 0) ? 0u : 1u);
            umma_f16_ts(tmem, acol + 64 + 8 * k, bd, GR_IDESC, 1u);
          }
          first = false;
          umma_commit(smem_u32(&vempty[vs]));
          umma_commit(smem_u32(&aempty[ab]));
        }
        if (!ok) break;
        umma_commit(smem_u32(accfull));
        ++nitem;
      }
      if (it > 0) mbar_wait(smem_u32(&aempty[(it - 1) & 1]), ((it - 1) >> 1) & 1, ws, nullptr);
    }
  } else {
    // ------------------------------------- scaling warps + epilogue -------
    const int sidx = tid - 64;           // 0..255
    const int quarter = warp & 3;        // TMEM lane quarter == channels 32 quarter .. +31
    const int th = (warp - 2) >> 2;      // token half of each tile (blocks 4 th .. 4 th + 3)
    const int m = quarter * 32 + lane;   // Gram row (channel) owned in the epilogue
    // ldmatrix row addresses: lane l -> matrix l / 8, row l % 8
    const int lm = lane >> 3, lr = lane & 7;
    uint32_t it = 0, nitem = 0;
    bool bad = false;
    Item item;
    for (int64_t i = blockIdx.x; decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
      asm volatile("bar.sync 1, 256;" ::: "memory");
      if ((sidx >> 5) < G) {  // scaler warp h computes head h's normaliser
        const int h = sidx >> 5;
        float M, Z;
        unit_softmax_stats_warp<G>(dm, ws, item.plane, item.seq, h, M, Z);
        if (lane == 0) {
          ustat[h] = M;
          ustat[G + h] = Z;
        }
      }
      asm volatile("bar.sync 1, 256;" ::: "memory");
      float us[2 * G];  // M_h, then 1/Z_h
#pragma unroll
      for (int e = 0; e < G; ++e) {
        us[e] = ustat[e];
        us[G + e] = 1.f / ustat[G + e];
      }
      // weights: thread pair (2 y2, 2 y2 + 1) shares token y2; thread `part`
      // sums heads part*NH .. part*NH + NH - 1 and one shuffle adds the halves
      constexpr int NH = G >= 2 ? G / 2 : 1;
      const int y2 = sidx >> 1, part = sidx & 1;
      const bool wact = G >= 2 || part == 0;
      const int h0 = G >= 2 ? part * NH : 0;
      float up[2 * NH];  // [M_h, then 1/Z_h] of this thread's heads (compile-time indices)
#pragma unroll
      for (int j = 0; j < NH; ++j) {
        up[j] = (G >= 2 && part) ? us[NH + j] : us[j];
        up[NH + j] = (G >= 2 && part) ? us[G + NH + j] : us[G + j];
      }
      float lc[NH], kc[NH];  // this thread's logits/kappa for the current tile
      const float* lkp = ws.lk + (int64_t)item.plane * dm.Ntot * (2 * G) + h0;
      if (wact && item.t0 + y2 < item.t1) load_lk_part<G, NH>(lkp + (item.t0 + y2) * (2 * G), lc, kc);

      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        const int vs = it % GR_VST, ab = it & 1;
        if (!mbar_wait(smem_u32(&vfull[vs]), (it / GR_VST) & 1, ws, abort)) goto scale_done;
        float* wt_s = wbuf + vs * TILE;
        {  // Eq. 8 weight of token t + y2
          const int64_t tok = t + y2;
          float ln[NH], kn[NH];
          if (wact && t + TILE + y2 < item.t1) load_lk_part<G, NH>(lkp + (t + TILE + y2) * (2 * G), ln, kn);
          float wp = 0.f;
          if (wact && tok < item.t1) wp = weight_part<NH, NH>(lc, kc, up, 0);
          const float wt = (wp + __shfl_xor_sync(0xffffffffu, wp, 1)) * dm.wdiv;
          if (part == 0 && tok < item.t1) {
            ws.w[(int64_t)item.plane * dm.Ntot + tok] = wt;
            bad |= !isfinite(wt);
          }
          if (part == 0) wt_s[y2] = tok < item.t1 ? wt : 0.f;
#pragma unroll
          for (int j = 0; j < NH; ++j) {
            lc[j] = ln[j];
            kc[j] = kn[j];
          }
        }
        asm volatile("bar.sync 1, 256;" ::: "memory");
        if (it >= 2 && !mbar_wait(smem_u32(&aempty[ab]), ((it >> 1) & 1) ^ 1, ws, abort)) goto scale_done;
        tc_fence_after();
        const uint32_t vt = smem_u32(vring + vs * GR_V_BYTES);
        const uint32_t acol = tmem + GR_ACOL + 128 * ab;
#pragma unroll
        for (int lh = 0; lh < 2; ++lh) {
          // one 32-column slab (this warp's 4 token blocks) of hi and of lo,
          // built in registers and written with one wide store each
          uint32_t hi[16], lo[16];
#pragma unroll
          for (int blk = 0; blk < 4; ++blk) {
            const int b = 4 * th + blk;  // 16-token block of the tile
            // weights of this thread's token pairs: rows 2(t%4), 2(t%4)+1 of each 8-token half
            const float2 wa = *(const float2*)(wt_s + 16 * b + 2 * (lane & 3));
            const float2 wb = *(const float2*)(wt_s + 16 * b + 8 + 2 * (lane & 3));
            // matrices: 0 = (tokens 0-7, ch c0..c0+7), 1 = (tokens 0-7, c0+8..), 2 = (8-15, c0..), 3 = (8-15, c0+8..)
            const int c0 = quarter * 32 + lh * 16 + (lm & 1) * 8;
            const int tokr = 16 * b + (lm >> 1) * 8 + lr;
            const uint32_t addr = vt + (c0 >> 6) * GR_BOX + sw128_off(tokr, (c0 & 63) >> 3);
            uint32_t r[4];
            ldsm_x4_trans(addr, r[0], r[1], r[2], r[3]);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              // x = w v (exact fp32 products), hi = bf16(x), lo = bf16(x - hi)
              const float2 x = __fmul2_rn(q < 2 ? wa : wb, make_float2(bf16lo(r[q]), bf16hi(r[q])));
              const uint32_t h = pack_bf16x2(x.x, x.y);
              const float2 res = __ffma2_rn(make_float2(bf16lo(h), bf16hi(h)), make_float2(-1.f, -1.f), x);
              // registers (r0 = lanes 0-7, r1 = lanes 8-15) of columns 8 blk + 4 (q / 2) ..
              hi[4 * blk + 2 * (q >> 1) + (q & 1)] = h;
              lo[4 * blk + 2 * (q >> 1) + (q & 1)] = pack_bf16x2(res.x, res.y);
            }
          }
          const uint32_t lanes = (uint32_t)(quarter * 32 + lh * 16) << 16;
          tmem_st_16x128b_x8(acol + lanes + 32 * th, hi);
          tmem_st_16x128b_x8(acol + lanes + 64 + 32 * th, lo);
        }
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&afull[ab]));
      }
      // epilogue: D is this chunk's partial Gram; warp (quarter, th) writes rows
      // 32 quarter .. +31, columns 64 th .. 64 th + 63
      if (!mbar_wait(smem_u32(accfull), nitem & 1, ws, abort)) goto scale_done;
      tc_fence_after();
      {
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16) + 64 * th;
        float* dst = ws.gpart + (((int64_t)item.plane * dm.c_cap + item.cidx) * D + m) * D + 64 * th;
#pragma unroll 1
        for (int cb = 0; cb < 2; ++cb) {
          float a[32];
          tmem_ld32(trow + cb * 32, a);
#pragma unroll
          for (int j = 0; j < 32; j += 4)
            *(float4*)(dst + cb * 32 + j) = make_float4(a[j], a[j + 1], a[j + 2], a[j + 3]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(accempty));
      ++nitem;
    }
  scale_done:
    if (bad) flag(ws, ST_NONFINITE);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, GR_TMEM_COLS);
  }
}

// ------------------------------------------------------------ SIMT fp32 ---
// float32 caches: thread t accumulates the 8x8 block (rows 8*(t/16), cols
// 8*(t%16)) of the chunk's partial Gram over 32-token slabs staged in SMEM.
constexpr int GF_THREADS = 256;
constexpr int GF_SLAB = 32;
constexpr int GF_LD = D + 4;

template <int G>
__global__ void __launch_bounds__(GF_THREADS)
    gram_f32_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu, const float* __restrict__ v) {
  __shared__ float xs[GF_SLAB][GF_LD];  // w_i v_i
  __shared__ float vs[GF_SLAB][GF_LD];  // v_i
  __shared__ float wsl[GF_SLAB];
  __shared__ float ustat[2 * G];
  __shared__ int s_skip;
  const int tid = threadIdx.x;
  if (tid == 0) s_skip = status_failed(ws) ? 1 : 0;
  __syncthreads();
  if (s_skip) return;
  const int rb = tid / 16, cb = tid % 16;
  bool bad = false;
  Item item;
  for (int64_t i = blockIdx.x; decode_item(dm, ws.plan, cu, i, item); i += gridDim.x) {
    const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
    const float* vbase = v + (int64_t)l * dm.kv_sl + (int64_t)g * dm.kv_sh;
    __syncthreads();
    if (tid < G) {
      float M, Z;
      unit_softmax_stats<G>(dm, ws, item.plane, item.seq, tid, M, Z);
      ustat[tid] = M;
      ustat[G + tid] = Z;
    }
    __syncthreads();
    float acc[8][8];
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
      for (int b = 0; b < 8; ++b) acc[a][b] = 0.f;
    for (int64_t t = item.t0; t < item.t1; t += GF_SLAB) {
      if (tid < GF_SLAB) {
        const int64_t tok = t + tid;
        float wt = 0.f;
        if (tok < item.t1) {
          wt = jacobian_weight<G>(dm, ws, ustat, item.plane, tok);
          ws.w[(int64_t)item.plane * dm.Ntot + tok] = wt;
          bad |= !isfinite(wt);
        }
        wsl[tid] = wt;
      }
      __syncthreads();
      for (int e = tid; e < GF_SLAB * (D / 4); e += GF_THREADS) {
        const int r = e / (D / 4), c4 = (e % (D / 4)) * 4;
        const int64_t tok = t + r;
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (tok < item.t1) x = *(const float4*)(vbase + tok * dm.kv_st + c4);
        const float wt = wsl[r];
        vs[r][c4] = x.x; vs[r][c4 + 1] = x.y; vs[r][c4 + 2] = x.z; vs[r][c4 + 3] = x.w;
        xs[r][c4] = wt * x.x; xs[r][c4 + 1] = wt * x.y; xs[r][c4 + 2] = wt * x.z; xs[r][c4 + 3] = wt * x.w;
      }
      __syncthreads();
#pragma unroll 4
      for (int r = 0; r < GF_SLAB; ++r) {
        float a[8], b[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          a[q] = vs[r][rb * 8 + q];
          b[q] = xs[r][cb * 8 + q];
        }
#pragma unroll
        for (int p = 0; p < 8; ++p)
#pragma unroll
          for (int q = 0; q < 8; ++q) acc[p][q] = fmaf(a[p], b[q], acc[p][q]);
      }
      __syncthreads();
    }
    float* dst = ws.gpart + ((int64_t)item.plane * dm.c_cap + item.cidx) * D * D;
#pragma unroll
    for (int p = 0; p < 8; ++p) {
      float* row = dst + (rb * 8 + p) * D + cb * 8;
      *(float4*)row = make_float4(acc[p][0], acc[p][1], acc[p][2], acc[p][3]);
      *(float4*)(row + 4) = make_float4(acc[p][4], acc[p][5], acc[p][6], acc[p][7]);
    }
  }
  if (bad) flag(ws, ST_NONFINITE);
}

// ------------------------------------------------------------ launchers ----
template <int G>
static cudaError_t launch_gram_g(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, int dtype, const void* v,
                                 const int32_t* cu, int grid, cudaStream_t st) {
  if (dtype == 1) {
    constexpr size_t smem = gram_bf16_smem_bytes();
    cudaError_t e =
        cudaFuncSetAttribute(gram_bf16_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    gram_bf16_kernel<G><<<grid, GR_THREADS, smem, st>>>(vmap, dm, ws, cu);
  } else {
    gram_f32_kernel<G><<<grid, GF_THREADS, 0, st>>>(dm, ws, cu, (const float*)v);
  }
  return cudaGetLastError();
}

cudaError_t launch_gram(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, int dtype, const void* v,
                        const int32_t* cu, int grid, cudaStream_t st) {
  switch (dm.G) {
    case 1: return launch_gram_g<1>(vmap, dm, ws, dtype, v, cu, grid, st);
    case 2: return launch_gram_g<2>(vmap, dm, ws, dtype, v, cu, grid, st);
    case 4: return launch_gram_g<4>(vmap, dm, ws, dtype, v, cu, grid, st);
    case 8: return launch_gram_g<8>(vmap, dm, ws, dtype, v, cu, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace jacap
