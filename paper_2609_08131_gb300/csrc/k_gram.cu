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
// bf16 caches use the 5th-generation tensor cores: A = V^T straight from the
// TMA-staged tile (bf16 is exact), B = [hi | lo] where w_i v_i = hi + lo is
// split into two bf16 halves by the scaling warps (residual error ~2^-17
// relative per product), so one kind::f16 MMA with N = 256 yields
// D[:, :128] + D[:, 128:] = sum_i v_i (w_i v_i)^T accumulated in fp32 in
// tensor memory. float32 caches take a SIMT fp32 kernel of the same contract.
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

template <int G>
__device__ __forceinline__ float jacobian_weight(const Dims& dm, const Ws& ws, const float* ustat, int plane,
                                                 int64_t tok) {
  const float* src = ws.lk + ((int64_t)plane * dm.Ntot + tok) * (2 * G);
  float lk[2 * G];
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
  float wt = 0.f;
#pragma unroll
  for (int h = 0; h < G; ++h) {
    const float a = expf(lk[h] - ustat[h]) / ustat[G + h];  // alpha_bar
    const float rho = a * (1.f - a);                           // diagonal of S
    wt = fmaf(rho * rho, lk[G + h], wt);                       // rho^2 kappa
  }
  return wt * dm.wdiv;
}

// --------------------------------------------------------------- tcgen05 ---
constexpr int GR_THREADS = 320;  // warp 0: TMA, warp 1: MMA, warps 2-9: scale + epilogue
constexpr int GR_SCALERS = 256;  // two threads per token row, interleaved 16-byte chunks
constexpr int GR_VST = 3;                     // V tiles in flight (TMA ring)
constexpr int GR_BST = 2;                     // hi/lo operand buffers
constexpr int GR_BOX = 16384;                 // {64 channels, 128 tokens} bf16, 128-byte swizzle
constexpr int GR_V_BYTES = 2 * GR_BOX;        // V tile
constexpr int GR_B_BYTES = 4 * GR_BOX;        // hi (2 boxes) + lo (2 boxes)
constexpr uint32_t GR_TMEM_COLS = 256;
// M = 128 (channels of V^T), N = 256 (hi | lo), both operands MN-major.
constexpr uint32_t GR_IDESC = idesc_bf16_f32(128, 256, 1, 1);

constexpr size_t gram_bf16_smem_bytes() { return 1024 + GR_VST * GR_V_BYTES + GR_BST * GR_B_BYTES + 256; }

template <int G>
__global__ void __launch_bounds__(GR_THREADS, 1)
    gram_bf16_kernel(const __grid_constant__ CUtensorMap vmap, Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* vring = smem;                                   // [GR_VST][GR_V_BYTES]
  uint8_t* bring = smem + GR_VST * GR_V_BYTES;             // [GR_BST][GR_B_BYTES]
  float* ustat = (float*)(bring + GR_BST * GR_B_BYTES);    // [2G] (<= 16 floats)
  uint64_t* vfull = (uint64_t*)(ustat + 16);
  uint64_t* vempty = vfull + GR_VST;
  uint64_t* bfull = vempty + GR_VST;
  uint64_t* bempty = bfull + GR_BST;
  uint64_t* accfull = bempty + GR_BST;
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
    for (int i = 0; i < GR_BST; ++i) {
      mbar_init(smem_u32(&bfull[i]), GR_SCALERS / 32);
      mbar_init(smem_u32(&bempty[i]), 1);
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
          const int vs = it % GR_VST, bs = it % GR_BST;
          if (!mbar_wait(smem_u32(&vfull[vs]), (it / GR_VST) & 1, ws, abort) ||
              !mbar_wait(smem_u32(&bfull[bs]), (it / GR_BST) & 1, ws, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t va = smem_u32(vring + vs * GR_V_BYTES);
          const uint32_t ba = smem_u32(bring + bs * GR_B_BYTES);
#pragma unroll
          for (int k = 0; k < TILE / 16; ++k) {  // 16 tokens per MMA
            const uint64_t ad = smem_desc_sw128(va + k * 2048, GR_BOX, 1024);
            const uint64_t bd = smem_desc_sw128(ba + k * 2048, GR_BOX, 1024);
            umma_f16_ss(tmem, ad, bd, GR_IDESC, (first && k == 0) ? 0u : 1u);
          }
          first = false;
          umma_commit(smem_u32(&vempty[vs]));
          umma_commit(smem_u32(&bempty[bs]));
        }
        if (!ok) break;
        umma_commit(smem_u32(accfull));
        ++nitem;
      }
    }
  } else {
    // ------------------------------------- scaling warps + epilogue -------
    const int sidx = tid - 64;                    // 0..255
    const int y = sidx >> 1;                      // token row 0..127 of each tile
    const int half = sidx & 1;                    // owns the 16-byte chunks cc with cc % 2 == half
    const int quarter = warp & 3;                 // TMEM lane quarter of this warp
    const int m = quarter * 32 + lane;            // Gram row (channel) owned in the epilogue
    const int colh = (warp - 2) >> 2;             // Gram columns [64 colh, 64 colh + 64) in the epilogue
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
      float us[2 * G];
#pragma unroll
      for (int e = 0; e < 2 * G; ++e) us[e] = ustat[e];
      float lkc[2 * G];  // logits/kappa of this thread's token in the current tile
      if (item.t0 + y < item.t1) load_lk<G>(dm, ws, item.plane, item.t0 + y, lkc);

      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        const int vs = it % GR_VST, bs = it % GR_BST;
        if (!mbar_wait(smem_u32(&vfull[vs]), (it / GR_VST) & 1, ws, abort)) goto scale_done;
        if (it >= (uint32_t)GR_BST && !mbar_wait(smem_u32(&bempty[bs]), ((it / GR_BST) & 1) ^ 1, ws, abort))
          goto scale_done;
        const int64_t tok = t + y;
        const bool valid = tok < item.t1;
        // logits/kappa of the next tile's token: issued now, used one tile later
        float lkn[2 * G];
        if (t + TILE + y < item.t1) load_lk<G>(dm, ws, item.plane, t + TILE + y, lkn);
        float wt = 0.f;
        if (valid) {
          wt = weight_from_lk<G>(dm, us, lkc);
          if (half == 0) {
            ws.w[(int64_t)item.plane * dm.Ntot + tok] = wt;
            bad |= !isfinite(wt);
          }
        }
#pragma unroll
        for (int e = 0; e < 2 * G; ++e) lkc[e] = lkn[e];
        const uint8_t* vt = vring + vs * GR_V_BYTES;
        uint8_t* bt = bring + bs * GR_B_BYTES;
        // half h owns box h (channels 64h..64h+63); at step q it takes 16-byte
        // chunk q ^ 4h, so the 8 lanes of each shared-memory phase (4 rows x 2
        // halves) touch 8 distinct bank groups under the 128-byte swizzle
        uint4 raw[8];
#pragma unroll
        for (int q = 0; q < 8; ++q)
          raw[q] = valid ? *(const uint4*)(vt + half * GR_BOX + sw128_off(y, q ^ (4 * half))) : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const uint32_t off = half * GR_BOX + sw128_off(y, q ^ (4 * half));
          const uint32_t rw[4] = {raw[q].x, raw[q].y, raw[q].z, raw[q].w};
          uint32_t hw[4], lw[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float x0 = wt * bf16lo(rw[e]);
            const float x1 = wt * bf16hi(rw[e]);
            hw[e] = pack_bf16x2(x0, x1);
            lw[e] = pack_bf16x2(x0 - bf16lo(hw[e]), x1 - bf16hi(hw[e]));
          }
          *(uint4*)(bt + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
          *(uint4*)(bt + 2 * GR_BOX + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&bfull[bs]));
      }
      // epilogue: D[:, :128] + D[:, 128:] is this chunk's partial Gram
      if (!mbar_wait(smem_u32(accfull), nitem & 1, ws, abort)) goto scale_done;
      tc_fence_after();
      {
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16) + 64 * colh;
        float* dst = ws.gpart + (((int64_t)item.plane * dm.c_cap + item.cidx) * D + m) * D + 64 * colh;
#pragma unroll 1
        for (int cb = 0; cb < 2; ++cb) {
          float a[32], b[32];
          tmem_ld32(trow + cb * 32, a);
          tmem_ld32(trow + 128 + cb * 32, b);
#pragma unroll
          for (int j = 0; j < 32; j += 4)
            *(float4*)(dst + cb * 32 + j) = make_float4(a[j] + b[j], a[j + 1] + b[j + 1], a[j + 2] + b[j + 2],
                                                        a[j + 3] + b[j + 3]);
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
