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
// tile (K-major), B = the group's G w centred queries, each split into a bf16
// hi and lo part (hi + lo is within 2^-18 relative of delta, so the centred
// logits carry about 17 significant bits of delta before fp32 accumulation
// instead of the 8 that one bf16 rounding would leave). The query-statistics
// kernel writes that B operand straight into the workspace in shared-memory
// image form; here it is one bulk copy per unit (a CTA's consecutive items
// of one unit share it), issued one item ahead into a double buffer. One MMA
// job of N = 2 rp columns per 128-token tile, the accumulator
// double-buffered in tensor memory, so one tile's readout overlaps
// the next tile's MMAs. Eight readout warps (two per tensor-memory lane
// quarter, alternating tiles) add the two parts, square and sum per head.
//
// Other shapes and float32 caches: a SIMT kernel (one thread per token, the
// tile's keys and one head's centred queries staged in shared memory).
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int KF_STAGES = 3;
constexpr int KF_BOX = 16384;  // {64 channels, 128 tokens} bf16
constexpr int KF_TILE_BYTES = 2 * KF_BOX;
constexpr int KF_THREADS = 320;  // warp 0: TMA, warp 1: MMA, warps 2-9: readout
constexpr int KF_READ0 = 2;
constexpr uint32_t KF_TMEM_COLS = 512;

template <int G, int W>
struct KfCfg {
  static constexpr int RP = kfull_rows_padded(G, W);  // padded rows per split part
  static constexpr int N = 2 * RP;                     // MMA N
  static constexpr int IMG_ATOM = N * 128;             // one 64-channel atom of the image
  static constexpr int IMG_BYTES = 2 * IMG_ATOM;       // = 512 RP, as written by the query statistics
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, N, 0, 0);
  static_assert(RP > 0 && N <= 256, "tensor-core shape");
  static constexpr size_t SMEM = 1024 + (size_t)KF_STAGES * KF_TILE_BYTES + 2 * (size_t)IMG_BYTES + 256;
};

template <int G, int W>
__global__ void __launch_bounds__(KF_THREADS, 1)
    kfull_bf16_kernel(const __grid_constant__ CUtensorMap kmap, Dims dm, Ws ws) {
  pdl_wait();
  using C = KfCfg<G, W>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tiles = smem;
  uint8_t* img = tiles + KF_STAGES * KF_TILE_BYTES;  // [2][IMG_BYTES]
  uint64_t* full = (uint64_t*)(img + 2 * C::IMG_BYTES);
  uint64_t* empty = full + KF_STAGES;
  uint64_t* accfull = empty + KF_STAGES;  // [2]
  uint64_t* accempty = accfull + 2;       // [2]
  uint64_t* imgfull = accempty + 2;       // [2]
  uint64_t* imgfree = imgfull + 2;        // [2]
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
      mbar_init(smem_u32(&imgfull[i]), 1);
      mbar_init(smem_u32(&imgfree[i]), 1);
    }
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
    // ------------------------------------ TMA: key tiles and query images --
    if (lane == 0) {
      prefetch_tmap(&kmap);
      auto issue_image = [&](const Item& item, uint32_t n) {
        const int p = n & 1;
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        const uint8_t* src = ws.qimg + (((int64_t)item.seq * dm.L + l) * dm.Hkv + g) * (int64_t)C::IMG_BYTES;
        mbar_arrive_expect_tx(smem_u32(&imgfull[p]), C::IMG_BYTES);
        bulk_g2s(smem_u32(img + p * C::IMG_BYTES), src, C::IMG_BYTES, smem_u32(&imgfull[p]));
      };
      uint32_t it = 0, nimg = 0;
      bool ok = true;
      ItemStream is(dm, ws, blockIdx.x, gridDim.x);
      Item cur, nxt;
      bool have = is.next(cur);
      if (have) issue_image(cur, nimg++);
      while (ok && have) {
        const int l = cur.plane / dm.Hkv, g = cur.plane % dm.Hkv;
        for (int64_t t = cur.t0; t < cur.t1; t += TILE) {
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
        if (!ok) break;
        // a next item of another unit needs its image: it goes to the buffer
        // of the run before this one, whose MMAs were all issued before this
        // run's first tile
        have = is.next(nxt);
        if (have) {
          if (nxt.plane != cur.plane || nxt.seq != cur.seq) {
            if (nimg >= 2 && !mbar_wait(smem_u32(&imgfree[nimg & 1]), ((nimg - 2) >> 1) & 1, ws, abort)) break;
            issue_image(nxt, nimg++);
          }
          cur = nxt;
        }
      }
      // no copy may still be landing when the CTA exits
      for (uint32_t k = (it > (uint32_t)KF_STAGES ? it - KF_STAGES : 0); k < it; ++k)
        mbar_wait(smem_u32(&full[k % KF_STAGES]), (k / KF_STAGES) & 1, ws, nullptr);
      for (uint32_t k = (nimg > 2u ? nimg - 2 : 0); k < nimg; ++k)
        mbar_wait(smem_u32(&imgfull[k & 1]), (k >> 1) & 1, ws, nullptr);
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer ----------
    if (lane == 0) {
      uint32_t it = 0, n = 0;  // n: runs (units) started
      bool ok = true, cont = false;
      int p = 0;
      Item item;
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        if (!cont) {
          p = n & 1;
          if (!mbar_wait(smem_u32(&imgfull[p]), (n >> 1) & 1, ws, abort)) break;
          tc_fence_after();
        }
        const uint64_t b0 = smem_desc_sw128(smem_u32(img + p * C::IMG_BYTES), 16, 1024);
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int st = it % KF_STAGES, slot = it & 1;
          if (!mbar_wait(smem_u32(&full[st]), (it / KF_STAGES) & 1, ws, abort) ||
              (it >= 2 && !mbar_wait(smem_u32(&accempty[slot]), ((it >> 1) & 1) ^ 1, ws, abort))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t a0 = smem_desc_sw128(smem_u32(tiles + st * KF_TILE_BYTES), 16, 1024);
          const uint32_t dacc = tmem + slot * 256;
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {  // descriptors advance by (byte offset >> 4)
            const uint64_t ad = a0 + (uint64_t)((((k >> 2) * KF_BOX) + (k & 3) * 32) >> 4);
            const uint64_t bd = b0 + (uint64_t)((((k >> 2) * C::IMG_ATOM) + (k & 3) * 32) >> 4);
            umma_f16_ss(dacc, ad, bd, C::IDESC, k > 0 ? 1u : 0u);
          }
          umma_commit(smem_u32(&accfull[slot]));
          umma_commit(smem_u32(&empty[st]));
        }
        if (!ok) break;
        cont = is.next_same_unit(item);
        if (!cont) {
          umma_commit(smem_u32(&imgfree[p]));
          ++n;
        }
      }
      // every MMA issued here completes before the CTA tears down tensor memory
      if (it > 0) mbar_wait(smem_u32(&accfull[(it - 1) & 1]), ((it - 1) >> 1) & 1, ws, nullptr);
    }
  } else {
    // ------------------------------------------------ readout -------------
    const int set = (warp - KF_READ0) >> 2;  // tiles with it % 2 == set
    const int quarter = warp & 3;
    const int y = quarter * 32 + lane;        // token row of the tile (tensor-memory lane)
    const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
    const float invw = 1.f / (float)(dm.cov_unbiased ? dm.window - 1 : dm.window);
    uint32_t it = 0;
    bool bad = false;
    Item item;
    for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
      float* lkp = ws.lk + (int64_t)item.plane * dm.Ntot * (2 * G) + G;
      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        if ((int)(it & 1) != set) continue;
        if (!mbar_wait(smem_u32(&accfull[set]), (it >> 1) & 1, ws, abort)) goto read_done;
        tc_fence_after();
        float kap[G];
#pragma unroll
        for (int hh = 0; hh < G; ++hh) kap[hh] = 0.f;
        const uint32_t ta = tmem + set * 256 + lanes;
#pragma unroll
        for (int b = 0; b < C::RP / 32; ++b) {
          uint32_t hi[32], lo[32];  // the two parts of 32 centred logits delta_j . k
          tmem_ld32x2(ta + b * 32, ta + C::RP + b * 32, hi, lo);
#pragma unroll
          for (int jj = 0; jj < 32; ++jj) {
            const int r = b * 32 + jj;
            if (r < G * W) {
              const float c = __uint_as_float(hi[jj]) + __uint_as_float(lo[jj]);
              kap[r / W] = fmaf(c, c, kap[r / W]);
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&accempty[set]));
        const int64_t tok = t + y;
        if (tok < item.t1) {
          float* dst = lkp + tok * (2 * G);
#pragma unroll
          for (int hh = 0; hh < G; ++hh) {
            const float v = kap[hh] * invw;
            bad |= !isfinite(v);
            dst[hh] = v;
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
  pdl_wait();
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
  JACAP_TRY(launch_pdl(dm.pdl != 0, kfull_bf16_kernel<G, W>, grid, KF_THREADS, C::SMEM, st, kmap, dm, ws));
  return cudaGetLastError();
}

template <int G>
static cudaError_t launch_kfull_g(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int grid, cudaStream_t st,
                                  bool* done) {
  *done = true;
  switch (dm.window) {
    case 8: if constexpr (kfull_rows_padded(G, 8) > 0) return launch_kfull_tc<G, 8>(kmap, dm, ws, grid, st); break;
    case 16: if constexpr (kfull_rows_padded(G, 16) > 0) return launch_kfull_tc<G, 16>(kmap, dm, ws, grid, st); break;
    case 32: if constexpr (kfull_rows_padded(G, 32) > 0) return launch_kfull_tc<G, 32>(kmap, dm, ws, grid, st); break;
    case 64: if constexpr (kfull_rows_padded(G, 64) > 0) return launch_kfull_tc<G, 64>(kmap, dm, ws, grid, st); break;
    default: break;
  }
  *done = false;
  return cudaSuccess;
}

// The tensor-core kernel reads the image that the query statistics wrote
// exactly when dm.kf_rp is set (bf16 cache and a supported shape).
bool kfull_uses_tensor_cores(const Dims& dm, int dtype) { return dtype == 1 && dm.kf_rp > 0; }

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
    JACAP_TRY(launch_pdl(dm.pdl != 0, kfull_simt_kernel<__nv_bfloat16>, grid, KS_THREADS, smem, st, dm, ws,
                         (const __nv_bfloat16*)k));
  } else {
    cudaError_t e =
        cudaFuncSetAttribute(kfull_simt_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    JACAP_TRY(launch_pdl(dm.pdl != 0, kfull_simt_kernel<float>, grid, KS_THREADS, smem, st, dm, ws, (const float*)k));
  }
  return cudaGetLastError();
}

}  // namespace jacap
