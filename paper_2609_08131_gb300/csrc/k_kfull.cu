// k_kfull.cu - kappa with the full window covariance of the queries.
//
// App. B.2 gives the O(N d^2) variant of the query-response variance,
//   kappa_h,i = k_i^T Lambda_h k_i,  Lambda_h = (1/w') sum_j delta_h,j delta_h,j^T,
// with delta_h,j = q_h,j - mu_h the centred window queries of head h and
// w' = w (or w - 1 with cov_unbiased). Since Lambda_h has rank <= w,
//   kappa_h,i = (1/w') sum_j (delta_h,j . k_i)^2,
// a contraction of every key with the G w centred queries followed by a sum of
// squares. These kernels run after the K pass (which supplies the logits and
// the softmax statistics) and overwrite its diagonal kappa.
//
// bf16 caches (w in {8, 16, 32, 64}, G w <= 128): tcgen05. A = the TMA-staged K
// tile (K-major), B = delta split exactly into three bf16 parts (hi + mid + lo
// carries ~24 significant bits; the centred logits then come out of the fp32
// accumulator without the error a single bf16 rounding of delta would leave).
// The heads are processed in jobs of g heads with g w <= 64, so a job's
// accumulator (3 blocks of RP = 32 or 64 columns) fits twice in tensor memory
// and one job's readout overlaps the next job's MMAs. Eight readout warps (two
// per tensor-memory lane quarter, alternating jobs) add the three parts,
// square and sum per head.
//
// Other shapes and float32 caches: a SIMT kernel (one thread per token, the
// tile's keys and one head's centred queries staged in shared memory).
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int KF_STAGES = 3;
constexpr int KF_BOX = 16384;  // {64 channels, 128 tokens} bf16
constexpr int KF_TILE_BYTES = 2 * KF_BOX;
constexpr int KF_THREADS = 448;  // warp 0: TMA, warp 1: MMA, warps 2-5: image, warps 6-13: readout
constexpr int KF_BUILD0 = 2, KF_READ0 = 6;
constexpr uint32_t KF_TMEM_COLS = 512;

template <int G, int W>
struct KfCfg {
  static constexpr int g = (G * W <= 64) ? G : 64 / W;   // heads per job
  static constexpr int ROWS = g * W;                        // delta rows per split part
  static constexpr int RP = ROWS <= 32 ? 32 : 64;           // padded rows per part
  static constexpr int N = 3 * RP;                          // MMA N
  static constexpr int NGR = G / g;                         // jobs per tile
  static constexpr int IMG_ATOM = N * 128;                  // one 64-channel atom of a job image
  static constexpr int JOB_BYTES = 2 * IMG_ATOM;
  static constexpr int IMG_BYTES = NGR * JOB_BYTES;
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, N, 0, 0);
  static_assert(G * W <= 128 && IMG_BYTES <= 96 * 1024, "image budget");
  static constexpr size_t SMEM = 1024 + (size_t)KF_STAGES * KF_TILE_BYTES + IMG_BYTES + 256;
};

template <int G, int W>
__global__ void __launch_bounds__(KF_THREADS, 1)
    kfull_bf16_kernel(const __grid_constant__ CUtensorMap kmap, Dims dm, Ws ws) {
  using C = KfCfg<G, W>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tiles = smem;
  uint8_t* img = tiles + KF_STAGES * KF_TILE_BYTES;
  uint64_t* full = (uint64_t*)(img + C::IMG_BYTES);
  uint64_t* empty = full + KF_STAGES;
  uint64_t* accfull = empty + KF_STAGES;  // [2]
  uint64_t* accempty = accfull + 2;       // [2]
  uint64_t* imgready = accempty + 2;
  uint64_t* imgfree = imgready + 1;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_skip;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_abort = 0;
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < KF_STAGES; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&accfull[i]), 1);
      mbar_init(smem_u32(&accempty[i]), 4);
    }
    mbar_init(smem_u32(imgready), 1);
    mbar_init(smem_u32(imgfree), 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (s_skip) return;
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), KF_TMEM_COLS);
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
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        for (int64_t t = item.t0; t < item.t1; t += TILE) {
          const int st = it % KF_STAGES;
          if (it >= (uint32_t)KF_STAGES &&
              !mbar_wait(smem_u32(&empty[st]), ((it / KF_STAGES) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          uint8_t* kt = tiles + st * KF_TILE_BYTES;
          mbar_arrive_expect_tx(smem_u32(&full[st]), KF_TILE_BYTES);
          tma_load_4d(smem_u32(kt), &kmap, 0, (int)t, g, l, smem_u32(&full[st]));
          tma_load_4d(smem_u32(kt + KF_BOX), &kmap, 64, (int)t, g, l, smem_u32(&full[st]));
          ++it;
        }
      }
      for (uint32_t k = (it > (uint32_t)KF_STAGES ? it - KF_STAGES : 0); k < it; ++k)
        mbar_wait(smem_u32(&full[k % KF_STAGES]), (k / KF_STAGES) & 1, ws, nullptr);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer ----------
    if (lane == 0) {
      uint32_t it = 0, nitem = 0, job = 0;
      bool ok = true;
      Item item;
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        if (!mbar_wait(smem_u32(imgready), nitem & 1, ws, abort)) break;
        tc_fence_after();
        const uint64_t b0 = smem_desc_sw128(smem_u32(img), 16, 1024);
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int st = it % KF_STAGES;
          if (!mbar_wait(smem_u32(&full[st]), (it / KF_STAGES) & 1, ws, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t a0 = smem_desc_sw128(smem_u32(tiles + st * KF_TILE_BYTES), 16, 1024);
#pragma unroll 1
          for (int grp = 0; grp < C::NGR; ++grp, ++job) {
            const int slot = job & 1;
            if (job >= 2 && !mbar_wait(smem_u32(&accempty[slot]), ((job >> 1) & 1) ^ 1, ws, abort)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t dacc = tmem + slot * 256;
#pragma unroll
            for (int k = 0; k < D / 16; ++k) {  // descriptors advance by (byte offset >> 4)
              const uint64_t ad = a0 + (uint64_t)((((k >> 2) * KF_BOX) + (k & 3) * 32) >> 4);
              const uint64_t bd =
                  b0 + (uint64_t)(((grp * C::JOB_BYTES) + ((k >> 2) * C::IMG_ATOM) + (k & 3) * 32) >> 4);
              umma_f16_ss(dacc, ad, bd, C::IDESC, k > 0 ? 1u : 0u);
            }
            umma_commit(smem_u32(&accfull[slot]));
          }
          if (!ok) break;
          umma_commit(smem_u32(&empty[st]));
        }
        if (!ok) break;
        umma_commit(smem_u32(imgfree));
        ++nitem;
      }
      // every MMA issued here completes before the CTA tears down tensor memory
      if (job > 0) mbar_wait(smem_u32(&accfull[(job - 1) & 1]), ((job - 1) >> 1) & 1, ws, nullptr);
    }
  } else if (warp < KF_READ0) {
    // ------------------------------ delta image, one item at a time -------
    // rows n = part * RP + r of job grp: r < ROWS holds part (hi, mid, lo) of
    // delta for head grp g + r / W, window query r % W; other rows are zero.
    // A failed wait (the abort flag is then set) still meets the builders'
    // barrier; all four builder warps leave together after it.
    const int bt = tid - 32 * KF_BUILD0;  // 0..127
    uint32_t nitem = 0;
    Item item;
    for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
      if (nitem > 0) mbar_wait(smem_u32(imgfree), (nitem - 1) & 1, ws, abort);
      named_barrier_sync(1, 128);
      if (*abort) break;
      const int l = item.plane / dm.Hkv, gkv = item.plane % dm.Hkv;
      const float* qd = ws.qdev + ((((int64_t)item.seq * dm.L + l) * dm.Hq + (int64_t)gkv * G) * dm.window) * D;
      for (int e = bt; e < C::NGR * C::N * 16; e += 128) {
        const int grp = e / (C::N * 16), rem = e % (C::N * 16);
        const int n = rem >> 4, cc = rem & 15;
        const int part = n / C::RP, r = n % C::RP;
        uint32_t wv[4] = {0u, 0u, 0u, 0u};
        if (r < C::ROWS) {
          const int hh = grp * C::g + r / W, j = r % W;
          const float* src = qd + ((int64_t)hh * dm.window + j) * D + cc * 8;
          const float4 x0 = *(const float4*)src, x1 = *(const float4*)(src + 4);
          const float xv[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            float y[2];
#pragma unroll
            for (int z = 0; z < 2; ++z) {
              const float v = xv[2 * q + z];
              const float hi = __bfloat162float(__float2bfloat16_rn(v));
              const float r1 = v - hi;
              const float mid = __bfloat162float(__float2bfloat16_rn(r1));
              y[z] = part == 0 ? hi : (part == 1 ? mid : r1 - mid);
            }
            wv[q] = pack_bf16x2(y[0], y[1]);
          }
        }
        *(uint4*)(img + grp * C::JOB_BYTES + (cc >> 3) * C::IMG_ATOM + sw128_off(n, cc & 7)) =
            make_uint4(wv[0], wv[1], wv[2], wv[3]);
      }
      fence_proxy_async_smem();
      named_barrier_sync(1, 128);
      if (bt == 0) mbar_arrive(smem_u32(imgready));
      ++nitem;
    }
  } else {
    // ------------------------------------------------ readout -------------
    const int set = (warp - KF_READ0) >> 2;   // jobs with job % 2 == set
    const int quarter = warp & 3;
    const int y = quarter * 32 + lane;         // token row of the tile (tensor-memory lane)
    const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
    const float invw = 1.f / (float)(dm.cov_unbiased ? dm.window - 1 : dm.window);
    uint32_t job = 0;
    bool bad = false;
    Item item;
    for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
      float* lkp = ws.lk + (int64_t)item.plane * dm.Ntot * (2 * G) + G;
      for (int64_t t = item.t0; t < item.t1; t += TILE) {
#pragma unroll 1
        for (int grp = 0; grp < C::NGR; ++grp, ++job) {
          if ((int)(job & 1) != set) continue;
          if (!mbar_wait(smem_u32(&accfull[set]), (job >> 1) & 1, ws, abort)) goto read_done;
          tc_fence_after();
          float kap[C::g];
#pragma unroll
          for (int hh = 0; hh < C::g; ++hh) kap[hh] = 0.f;
          const uint32_t ta = tmem + set * 256 + lanes;
#pragma unroll
          for (int b = 0; b < C::RP / 32; ++b) {
            float c[32], p[32];  // c: centred logits delta_j . k, the three parts added
            tmem_ld32(ta + b * 32, c);
#pragma unroll
            for (int part = 1; part < 3; ++part) {
              tmem_ld32(ta + part * C::RP + b * 32, p);
#pragma unroll
              for (int jj = 0; jj < 32; ++jj) c[jj] += p[jj];
            }
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
              const int r = b * 32 + jj;
              if (r < C::ROWS) kap[r / W] = fmaf(c[jj], c[jj], kap[r / W]);
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&accempty[set]));
          const int64_t tok = t + y;
          if (tok < item.t1) {
            float* dst = lkp + tok * (2 * G) + grp * C::g;
#pragma unroll
            for (int hh = 0; hh < C::g; ++hh) {
              const float v = kap[hh] * invw;
              bad |= !isfinite(v);
              dst[hh] = v;
            }
          }
        }
      }
    }
  read_done:
    if (bad) flag(ws, ST_NONFINITE);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, KF_TMEM_COLS);
  }
}

// ------------------------------------------------------------ SIMT ---------
constexpr int KS_THREADS = 128;
constexpr int KS_LD = D + 1;
constexpr int KS_WMAX = 64;  // window queries staged per round

template <typename T>
__global__ void __launch_bounds__(KS_THREADS)
    kfull_simt_kernel(Dims dm, Ws ws, const T* __restrict__ k) {
  extern __shared__ float ksm[];
  float* Ks = ksm;                    // [TILE][KS_LD] the tile's keys
  float* Qs = ksm + TILE * KS_LD;     // [KS_WMAX][D] centred queries of one head
  __shared__ int s_skip;
  const int tid = threadIdx.x;
  if (tid == 0) s_skip = status_failed(ws) ? 1 : 0;
  __syncthreads();
  if (s_skip) return;
  const int G = dm.G;
  const float invw = 1.f / (float)(dm.cov_unbiased ? dm.window - 1 : dm.window);
  bool bad = false;
  Item item;
  for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
    const int l = item.plane / dm.Hkv, gkv = item.plane % dm.Hkv;
    const T* kb = k + (int64_t)l * dm.kv_sl + (int64_t)gkv * dm.kv_sh;
    for (int64_t t = item.t0; t < item.t1; t += TILE) {
      __syncthreads();
      for (int e = tid; e < TILE * D; e += KS_THREADS) {
        const int r = e / D, c = e % D;
        Ks[r * KS_LD + c] = (t + r < item.t1) ? (float)kb[(t + r) * dm.kv_st + c] : 0.f;
      }
      for (int hh = 0; hh < G; ++hh) {
        const float* qd =
            ws.qdev + ((((int64_t)item.seq * dm.L + l) * dm.Hq + (int64_t)gkv * G + hh) * dm.window) * D;
        float kap = 0.f;
        for (int j0 = 0; j0 < dm.window; j0 += KS_WMAX) {
          const int nj = min(KS_WMAX, dm.window - j0);
          __syncthreads();
          for (int e = tid; e < nj * D; e += KS_THREADS) Qs[e] = qd[(int64_t)j0 * D + e];
          __syncthreads();
          for (int j = 0; j < nj; ++j) {
            float c = 0.f;
            for (int ch = 0; ch < D; ++ch) c = fmaf(Qs[j * D + ch], Ks[tid * KS_LD + ch], c);
            kap = fmaf(c, c, kap);
          }
        }
        const int64_t tok = t + tid;
        if (tok < item.t1) {
          const float v = kap * invw;
          bad |= !isfinite(v);
          ws.lk[((int64_t)item.plane * dm.Ntot + tok) * (2 * G) + G + hh] = v;
        }
      }
    }
  }
  if (bad) flag(ws, ST_NONFINITE);
}

// ------------------------------------------------------------ launchers ----
template <int G, int W>
static cudaError_t launch_kfull_tc(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int grid, cudaStream_t st) {
  using C = KfCfg<G, W>;
  static_assert(C::SMEM <= 232448, "shared memory budget");
  cudaError_t e =
      cudaFuncSetAttribute(kfull_bf16_kernel<G, W>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  if (e != cudaSuccess) return e;
  kfull_bf16_kernel<G, W><<<grid, KF_THREADS, C::SMEM, st>>>(kmap, dm, ws);
  return cudaGetLastError();
}

template <int G>
static cudaError_t launch_kfull_g(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int grid, cudaStream_t st,
                                  bool* done) {
  *done = true;
  switch (dm.window) {
    case 8: if constexpr (G * 8 <= 128) return launch_kfull_tc<G, 8>(kmap, dm, ws, grid, st); break;
    case 16: if constexpr (G * 16 <= 128) return launch_kfull_tc<G, 16>(kmap, dm, ws, grid, st); break;
    case 32: if constexpr (G * 32 <= 128) return launch_kfull_tc<G, 32>(kmap, dm, ws, grid, st); break;
    case 64: if constexpr (G * 64 <= 128) return launch_kfull_tc<G, 64>(kmap, dm, ws, grid, st); break;
    default: break;
  }
  *done = false;
  return cudaSuccess;
}

bool kfull_uses_tensor_cores(const Dims& dm, int dtype) {
  if (dtype != 1) return false;
  const int w = dm.window;
  return (w == 8 || w == 16 || w == 32 || w == 64) && dm.G * w <= 128;
}

cudaError_t launch_kfull(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int dtype, const void* k, int grid,
                         cudaStream_t st) {
  if (kfull_uses_tensor_cores(dm, dtype)) {
    bool done = false;
    cudaError_t e = cudaSuccess;
    switch (dm.G) {
      case 1: e = launch_kfull_g<1>(kmap, dm, ws, grid, st, &done); break;
      case 2: e = launch_kfull_g<2>(kmap, dm, ws, grid, st, &done); break;
      case 4: e = launch_kfull_g<4>(kmap, dm, ws, grid, st, &done); break;
      case 8: e = launch_kfull_g<8>(kmap, dm, ws, grid, st, &done); break;
      default: break;
    }
    if (done) return e;
  }
  constexpr size_t smem = (size_t)(TILE * KS_LD + KS_WMAX * D) * sizeof(float);
  if (dtype == 1) {
    cudaError_t e = cudaFuncSetAttribute(kfull_simt_kernel<__nv_bfloat16>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kfull_simt_kernel<__nv_bfloat16><<<grid, KS_THREADS, smem, st>>>(dm, ws, (const __nv_bfloat16*)k);
  } else {
    cudaError_t e =
        cudaFuncSetAttribute(kfull_simt_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kfull_simt_kernel<float><<<grid, KS_THREADS, smem, st>>>(dm, ws, (const float*)k);
  }
  return cudaGetLastError();
}

}  // namespace jacap
