// k_stream.cu - work plan, query-window statistics and the streaming K pass.
//
//  plan_kernel          clears the status word, validates cu_seqlens and lays
//                       out the work items (chunks of `chunk` tokens that never
//                       straddle requests) in the chunk table.
//  window_stats_kernel  mu_h and the diagonal of Lambda_Q from the last w queries
//                       of each query head (Sec. 3.4 last paragraph; App. B.2).
//  kpass_kernel         (float32 caches; bf16 caches use k_kpass.cu) one
//                       streaming pass over K with TMA-staged 128-token
//                       tiles: for each token and each query head h of its group
//                       the pool logit l = k.mu_h/(tau sqrt d) (Sec. 3.4, Alg. 1
//                       step 1) and kappa = sum_c lambda_h,c k_c^2 (Sec. 3.4),
//                       plus an online (max, sum exp) per chunk and head that the
//                       next pass combines into the softmax normaliser.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

// The pass's first kernel, one block: clears the status word, validates
// cu_seqlens and lays out the chunks (thread 0), then writes the chunk table:
// record r = {t0, t1, request, r} for the C_tot chunks of a plane.
__global__ void __launch_bounds__(256) plan_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  pdl_wait();
  __shared__ int s_ctot;
  if (threadIdx.x < 16) ws.status[threadIdx.x] = 0u;
  if (threadIdx.x == 0) {
    bool ok = (cu[0] == 0) && ((int64_t)cu[dm.S] == dm.Ntot);
    int32_t acc = 0;
    ws.plan[1] = 0;
    for (int s = 0; s < dm.S; ++s) {
      const int32_t n = cu[s + 1] - cu[s];
      if (n < 0) ok = false;
      const int32_t c = n > 0 ? (n + dm.chunk - 1) / dm.chunk : 0;
      acc += c;
      ws.plan[2 + s] = acc;
    }
    if (!ok || acc > dm.c_cap) {
      atomicOr(ws.status, ST_INVALID);
      acc = 0;
    }
    ws.plan[0] = acc;
    s_ctot = acc;
  }
  // the fused schedule's per-unit progress counters (gcount, then fdone)
  const int64_t units = (int64_t)dm.L * dm.Hkv * dm.S;
  for (int64_t i = threadIdx.x; i < 2 * units; i += blockDim.x) ws.gcount[i] = 0;
#ifdef JACAP_TRACE
  if (ws.trace != nullptr)
    for (int64_t i = threadIdx.x; i < TR_SLOTS * units; i += blockDim.x)
      ws.trace[i] = (i % TR_SLOTS == TR_GRAM0 || i % TR_SLOTS == TR_SC_IMG || i % TR_SLOTS == TR_SC_MMA) ? ~0ull : 0ull;
  if (ws.trace_cta != nullptr)
    for (int64_t i = threadIdx.x; i < (int64_t)TR_KERNELS * TR_CTAS * TR_CTA_SLOTS; i += blockDim.x) ws.trace_cta[i] = 0;
#endif
  __syncthreads();
  const int ctot = s_ctot;
  for (int r = threadIdx.x; r < ctot; r += blockDim.x) {
    // largest s with prefix[s] <= r (prefix is plan[1 .. S+1], nondecreasing)
    int lo = 0, hi = dm.S - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (ws.plan[1 + mid] <= r) lo = mid; else hi = mid - 1;
    }
    const int64_t t0 = (int64_t)cu[lo] + (int64_t)(r - ws.plan[1 + lo]) * dm.chunk;
    const int64_t t1 = min((int64_t)cu[lo + 1], t0 + (int64_t)dm.chunk);
    ws.chunks[r] = make_int4((int)t0, (int)t1, lo, r);
  }
}

template <typename T>
__device__ __forceinline__ float ld_elem(const T* p);
template <>
__device__ __forceinline__ float ld_elem<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float ld_elem<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}

// Self-test of the bounded waits: one thread waits on an mbarrier that nothing
// arrives on, with the wait code every pipeline of the pass uses but a short
// limit; on expiry it sets ST_TIMEOUT in the status word (cleared first) and
// returns. Nothing faults and the context stays usable.
__global__ void __launch_bounds__(32) selftest_wait_kernel(Ws ws, unsigned long long limit_ns) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    for (int i = 0; i < 16; ++i) ws.status[i] = 0u;
    mbar_init(smem_u32(&bar), 1);
    fence_mbar_init();
  }
  __syncwarp();
  if (threadIdx.x == 0) mbar_wait_slow(smem_u32(&bar), 0, ws, nullptr, limit_ns);  // phase 0 never completes
}

cudaError_t launch_selftest_wait(const Ws& ws, unsigned long long limit_ns, cudaStream_t st) {
  selftest_wait_kernel<<<1, 32, 0, st>>>(ws, limit_ns);
  return cudaGetLastError();
}

// One block per (request, layer, query head); thread c owns channel c.
template <typename T>
__global__ void __launch_bounds__(D) window_stats_kernel(Dims dm, Ws ws, const T* __restrict__ q) {
  pdl_wait();
  if (status_failed(ws)) return;
  const int b = blockIdx.x;
  const int h = b % dm.Hq;
  const int l = (b / dm.Hq) % dm.L;
  const int s = b / (dm.Hq * dm.L);
  const int c = threadIdx.x;
  const T* base = q + (int64_t)s * dm.q_ss + (int64_t)l * dm.q_sl + (int64_t)h * dm.q_sh + c;
  float sum = 0.f;
  for (int j = 0; j < dm.window; ++j) sum += ld_elem(base + (int64_t)j * dm.q_sp);
  const float mu = sum / (float)dm.window;
  float ss = 0.f;
  for (int j = 0; j < dm.window; ++j) {
    const float e = ld_elem(base + (int64_t)j * dm.q_sp) - mu;
    ss = fmaf(e, e, ss);
  }
  const float lam = ss / (float)(dm.cov_unbiased ? dm.window - 1 : dm.window);
  const int64_t o = (((int64_t)s * dm.L + l) * dm.Hq + h) * D + c;
  if (dm.full_cov && dm.kf_rp) {
    // centred window queries as the B operand image of the full-covariance
    // MMA (K-major, 128-byte swizzle, two 64-channel atoms of 2 rp rows): row
    // r = hh W + j holds the bf16 rounding hi of q_j - mu, row rp + r the
    // bf16 rounding of the remainder, so hi + lo is within 2^-18 of q_j - mu
    const int rp = dm.kf_rp, hh = h % dm.G;
    uint8_t* img = ws.qimg + (((int64_t)s * dm.L + l) * dm.Hkv + h / dm.G) * (int64_t)(512 * rp);
    img += (c >> 6) * (256 * rp) + (c & 7) * 2;
    const uint32_t chunk = (c & 63) >> 3;
    for (int j = 0; j < dm.window; ++j) {
      const float e = ld_elem(base + (int64_t)j * dm.q_sp) - mu;
      const __nv_bfloat16 hi = __float2bfloat16_rn(e);
      const uint32_t r = (uint32_t)(hh * dm.window + j);
      *(__nv_bfloat16*)(img + sw128_off(r, chunk)) = hi;
      *(__nv_bfloat16*)(img + sw128_off(rp + r, chunk)) = __float2bfloat16_rn(e - __bfloat162float(hi));
    }
    if (hh == 0)  // padding rows of the group
      for (int r = dm.G * dm.window; r < rp; ++r) {
        *(__nv_bfloat16*)(img + sw128_off(r, chunk)) = __float2bfloat16_rn(0.f);
        *(__nv_bfloat16*)(img + sw128_off(rp + r, chunk)) = __float2bfloat16_rn(0.f);
      }
  } else if (dm.full_cov) {  // fp32 centred window queries for the CUDA-core kernel
    float* dst = ws.qdev + ((((int64_t)s * dm.L + l) * dm.Hq + h) * dm.window) * D + c;
    for (int j = 0; j < dm.window; ++j) dst[(int64_t)j * D] = ld_elem(base + (int64_t)j * dm.q_sp) - mu;
  }
  ws.mu[o] = mu * dm.inv_scale;
  ws.lam[o] = lam;
  if (!isfinite(mu) || !isfinite(lam)) flag(ws, ST_NONFINITE);
}

// ------------------------------------------------------------------ K pass --
// Warps 0-3: one thread per token of the current tile; warp 4: TMA producer.
constexpr int KP_THREADS = 160;

template <typename T>
struct KpCfg {
  static constexpr int ES = sizeof(T);
  static constexpr int BOX_C = 128 / ES;           // channels per 128-byte box row
  static constexpr int NBOX = D / BOX_C;           // boxes per tile row
  static constexpr int BOX_BYTES = TILE * 128;     // 16 KB
  static constexpr int TILE_BYTES = NBOX * BOX_BYTES;
  static constexpr int STAGES = (ES == 2) ? 4 : 3;
};

template <typename T, int G>
constexpr size_t kpass_smem_bytes() {
  return 1024 /*align slack*/ + (size_t)KpCfg<T>::STAGES * KpCfg<T>::TILE_BYTES + 2 * G * D * 4 +
         2 * G * 128 * 4 + 2 * KpCfg<T>::STAGES * 8 + 64;
}

template <typename T, int G>
__global__ void __launch_bounds__(KP_THREADS, 1)
    kpass_kernel(const __grid_constant__ CUtensorMap kmap, Dims dm, Ws ws, const int32_t* __restrict__ cu) {
  pdl_wait();
  using C = KpCfg<T>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tiles = smem;
  float* mu_s = (float*)(tiles + C::STAGES * C::TILE_BYTES);
  float* lam_s = mu_s + G * D;
  float* red = lam_s + G * D;  // [2G][128]
  uint64_t* full = (uint64_t*)(red + 2 * G * 128);
  uint64_t* empty = full + C::STAGES;
  __shared__ int s_abort;
  __shared__ int s_skip;

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_abort = 0;
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < C::STAGES; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 4);
    }
    fence_mbar_init();
  }
  __syncthreads();
  if (s_skip) return;
  volatile int* abort = &s_abort;

  if (warp == 4) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      prefetch_tmap(&kmap);
      uint32_t it = 0;
      bool ok = true;
      Item item;
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        for (int64_t t = item.t0; t < item.t1; t += TILE) {
          const int st = it % C::STAGES;
          if (it >= (uint32_t)C::STAGES &&
              !mbar_wait(smem_u32(&empty[st]), ((it / C::STAGES) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(smem_u32(&full[st]), C::TILE_BYTES);
#pragma unroll
          for (int b = 0; b < C::NBOX; ++b)
            tma_load_4d(smem_u32(tiles + st * C::TILE_BYTES + b * C::BOX_BYTES), &kmap, b * C::BOX_C, (int)t, g,
                        l, smem_u32(&full[st]));
          ++it;
        }
      }
      // Drain: every copy issued into a stage has landed before the CTA can
      // exit (returns at once on the normal path, bounded after an abort).
      for (uint32_t k = (it > (uint32_t)C::STAGES ? it - C::STAGES : 0); k < it; ++k)
        mbar_wait(smem_u32(&full[k % C::STAGES]), (k / C::STAGES) & 1, ws, nullptr);
    }
    return;
  }

  // ---------------- compute warps: thread y owns row y of each tile ----------
  const int y = tid;  // 0..127
  uint32_t it = 0;
  bool bad = false;
  Item item;
  for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
    const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
    // query statistics of the G heads of this KV head
    asm volatile("bar.sync 1, 128;" ::: "memory");
    {
      const int64_t qbase = (((int64_t)item.seq * dm.L + l) * dm.Hq + (int64_t)g * G) * D;
      for (int e = y; e < G * D; e += 128) {
        mu_s[e] = ws.mu[qbase + e];
        lam_s[e] = ws.lam[qbase + e];
      }
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");

    float run_m[G], run_s[G];
#pragma unroll
    for (int h = 0; h < G; ++h) {
      run_m[h] = -INFINITY;
      run_s[h] = 0.f;
    }
    for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
      const int st = it % C::STAGES;
      if (!mbar_wait(smem_u32(&full[st]), (it / C::STAGES) & 1, ws, abort)) goto compute_done;
      const uint8_t* tile = tiles + st * C::TILE_BYTES;
      float2 lacc[G], kacc[G];
#pragma unroll
      for (int h = 0; h < G; ++h) {
        lacc[h] = make_float2(0.f, 0.f);
        kacc[h] = make_float2(0.f, 0.f);
      }
#pragma unroll 2
      for (int cc = 0; cc < D * C::ES / 16; ++cc) {  // 16-byte chunks of the row
        const int b = cc >> 3, ch = cc & 7;
        const uint4 raw = *(const uint4*)(tile + b * C::BOX_BYTES + sw128_off(y, ch));
        float kv[8];
        constexpr int NV = 16 / C::ES;  // values in the chunk: 8 (bf16) or 4 (f32)
        if constexpr (C::ES == 2) {
          kv[0] = bf16lo(raw.x); kv[1] = bf16hi(raw.x);
          kv[2] = bf16lo(raw.y); kv[3] = bf16hi(raw.y);
          kv[4] = bf16lo(raw.z); kv[5] = bf16hi(raw.z);
          kv[6] = bf16lo(raw.w); kv[7] = bf16hi(raw.w);
        } else {
          kv[0] = __uint_as_float(raw.x); kv[1] = __uint_as_float(raw.y);
          kv[2] = __uint_as_float(raw.z); kv[3] = __uint_as_float(raw.w);
        }
        const int c0 = cc * NV;
#pragma unroll
        for (int p = 0; p < NV / 2; ++p) {
          const float2 kk = make_float2(kv[2 * p], kv[2 * p + 1]);
          const float2 sq = __fmul2_rn(kk, kk);
#pragma unroll
          for (int h = 0; h < G; ++h) {
            const float2 m = *(const float2*)(mu_s + h * D + c0 + 2 * p);
            const float2 a = *(const float2*)(lam_s + h * D + c0 + 2 * p);
            lacc[h] = __ffma2_rn(kk, m, lacc[h]);
            kacc[h] = __ffma2_rn(sq, a, kacc[h]);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&empty[st]));

      const int64_t tok = t + y;
      if (tok < item.t1) {
        float out[2 * G];
#pragma unroll
        for (int h = 0; h < G; ++h) {
          const float lg = lacc[h].x + lacc[h].y;
          const float kp = kacc[h].x + kacc[h].y;
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
        store_floats<2 * G, LkAlign<G>::ROW>(dst, out);
      }
    }
    // chunk statistics: combine the 128 per-thread (max, sum) pairs per head
#pragma unroll
    for (int h = 0; h < G; ++h) {
      red[h * 128 + y] = run_m[h];
      red[(G + h) * 128 + y] = run_s[h];
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (y < G) {
      const int h = y;
      float m = -INFINITY;
      for (int j = 0; j < 128; ++j) m = fmaxf(m, red[h * 128 + j]);
      float ssum = 0.f;
      for (int j = 0; j < 128; ++j) {
        const float mj = red[h * 128 + j];
        if (mj > -INFINITY) ssum += red[(G + h) * 128 + j] * expf(mj - m);
      }
      float* cs = ws.cstats + (((int64_t)item.plane * dm.c_cap + item.cidx) * G + h) * 2;
      cs[0] = m;
      cs[1] = ssum;
    }
  }
compute_done:
  if (bad) flag(ws, ST_NONFINITE);
}

// ------------------------------------------------------------ launchers ----
template <typename T>
static cudaError_t launch_window_stats_t(const Dims& dm, const Ws& ws, const void* q, cudaStream_t st) {
  const int blocks = dm.S * dm.L * dm.Hq;
  JACAP_TRY(launch_pdl(dm.pdl != 0, window_stats_kernel<T>, blocks, D, 0, st, dm, ws, (const T*)q));
  return cudaGetLastError();
}

cudaError_t launch_plan(const Dims& dm, const Ws& ws, const int32_t* cu, cudaStream_t st) {
  JACAP_TRY(launch_pdl(dm.pdl != 0, plan_kernel, 1, 256, 0, st, dm, ws, cu));
  return cudaGetLastError();
}

cudaError_t launch_window_stats(const Dims& dm, const Ws& ws, int dtype, const void* q, cudaStream_t st) {
  return dtype == 1 ? launch_window_stats_t<__nv_bfloat16>(dm, ws, q, st)
                    : launch_window_stats_t<float>(dm, ws, q, st);
}

template <typename T, int G>
static cudaError_t launch_kpass_tg(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, const int32_t* cu,
                                   int grid, cudaStream_t st) {
  constexpr size_t smem = kpass_smem_bytes<T, G>();
  cudaError_t e = cudaFuncSetAttribute(kpass_kernel<T, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  JACAP_TRY(launch_pdl(dm.pdl != 0, kpass_kernel<T, G>, grid, KP_THREADS, smem, st, kmap, dm, ws, cu));
  return cudaGetLastError();
}

template <typename T>
static cudaError_t launch_kpass_t(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, const int32_t* cu,
                                  int grid, cudaStream_t st) {
  switch (dm.G) {
    case 1: return launch_kpass_tg<T, 1>(kmap, dm, ws, cu, grid, st);
    case 2: return launch_kpass_tg<T, 2>(kmap, dm, ws, cu, grid, st);
    case 3: return launch_kpass_tg<T, 3>(kmap, dm, ws, cu, grid, st);
    case 4: return launch_kpass_tg<T, 4>(kmap, dm, ws, cu, grid, st);
    case 5: return launch_kpass_tg<T, 5>(kmap, dm, ws, cu, grid, st);
    case 6: return launch_kpass_tg<T, 6>(kmap, dm, ws, cu, grid, st);
    case 7: return launch_kpass_tg<T, 7>(kmap, dm, ws, cu, grid, st);
    case 8: return launch_kpass_tg<T, 8>(kmap, dm, ws, cu, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_kpass(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int dtype, const int32_t* cu,
                         int grid, cudaStream_t st) {
  // bf16: logits on the tensor cores (k_kpass.cu); float32: the SIMT pass above
  return dtype == 1 ? launch_kpass_bf16(kmap, dm, ws, cu, grid, st) : launch_kpass_t<float>(kmap, dm, ws, cu, grid, st);
}

}  // namespace jacap
