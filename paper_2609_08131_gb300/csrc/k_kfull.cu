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
// bf16 caches (w in {8, 16, 32, 64}, G w <= 128): one tcgen05 kernel does the
// whole K pass in this mode, so K is read once: the pool-softmax logits
// l_h = k . mu'_h (mu' = mu / (tau sqrt d)), this kappa and the per-chunk
// softmax statistics. A = the TMA-staged K tile (K-major); B = a per-unit
// image with, per 64-channel atom, two sections of N = rp + nb rows:
//   section 0: rows 0 .. rp-1   hi(delta_j), the bf16 rounding of q_j - mu,
//              rows rp .. rp+nb-1  mu' split exactly into three bf16 parts;
//   section 1: rows 0 .. rp-1   lo(delta_j), the bf16 rounding of the rest,
//              rows rp .. rp+nb-1  zero.
// Two MMAs of N columns per 16 channels accumulate both sections into one
// accumulator, so column j < rp holds delta_j . k with hi + lo within 2^-18
// relative of delta (about 17 significant bits before fp32 accumulation
// instead of the 8 that one bf16 rounding would leave), and column rp + n
// part n of mu' . k. The query-statistics kernel writes the delta rows in
// image form into the workspace; here they arrive by bulk copies, once per
// run of a CTA's consecutive items of one unit, and a builder warp adds the
// mu' rows. Four readout warps (one per tensor-memory lane quarter) square and
// sum the delta columns per head, add the three logit parts, keep the online
// (max, sum exp) and write the token's logits/kappa row in one piece.
//
// Other shapes and float32 caches: a SIMT kernel (one thread per token, the
// tile's keys and one head's centred queries staged in shared memory).
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int KX_STAGES = 4;
constexpr int KX_BOX = 16384;  // {64 channels, 128 tokens} bf16
constexpr int KX_TILE_BYTES = 2 * KX_BOX;
constexpr int KX_THREADS = 256;  // warp 0: TMA, 1: MMA, 2: image builder, 3: idle, 4-7: readout
constexpr int KX_READ0 = 4;
constexpr uint32_t KX_TMEM_COLS = 512;

template <int G, int W>
struct KxCfg {
  static constexpr int RP = kfull_rows_padded(G, W);  // delta rows (G w, padded)
  static constexpr int NB = (3 * G <= 16) ? 16 : 32;   // mu' rows (3 G parts, padded)
  static constexpr int N = RP + NB;                    // MMA N
  static constexpr int SEC = N * 128;                  // bytes of one section of one atom
  static constexpr int ATOM = 2 * SEC;
  static constexpr int IMG_BYTES = 2 * ATOM;
  static constexpr int QIMG_BYTES = 512 * RP;          // the delta image as the query statistics write it
  static constexpr uint32_t ACC = N <= 128 ? 128 : 256;  // tensor-memory columns per accumulator
  static constexpr uint32_t IDESC = idesc_bf16_f32(128, N, 0, 0);
  static_assert(RP > 0 && N <= 256 && N % 16 == 0 && 2 * ACC <= KX_TMEM_COLS, "tensor-core shape");
  static_assert(SEC % 1024 == 0, "sections start on a swizzle-pattern boundary");
  static constexpr size_t SMEM = 1024 + (size_t)KX_STAGES * KX_TILE_BYTES + IMG_BYTES + 4 * 2 * G * 4 + 256;
};

// Rows rp .. rp + nb - 1 of section 0 of both atoms: row rp + part G + h holds
// part (0 hi, 1 mid, 2 lo) of mu'_h with hi + mid + lo = mu'_h to about 24
// bits; rows past 3 G are zero. One warp.
template <int G, int W>
__device__ __forceinline__ void write_mu_rows(uint8_t* img, const float* mu, int lane) {
  using C = KxCfg<G, W>;
  for (int e = lane; e < C::NB * 16; e += 32) {
    const int n = e >> 4, cc = e & 15;  // row, 8-channel chunk
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
    *(uint4*)(img + (cc >> 3) * C::ATOM + sw128_off(C::RP + n, cc & 7)) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  }
}

template <int G, int W>
__global__ void __launch_bounds__(KX_THREADS, 1)
    kpass_full_bf16_kernel(const __grid_constant__ CUtensorMap kmap, Dims dm, Ws ws) {
  pdl_wait();
  using C = KxCfg<G, W>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
  uint8_t* tiles = smem;
  uint8_t* img = tiles + KX_STAGES * KX_TILE_BYTES;     // one image, refilled per run
  float* red = (float*)(img + C::IMG_BYTES);             // [4 readout warps][2G]
  uint64_t* full = (uint64_t*)(red + 4 * 2 * G);
  uint64_t* empty = full + KX_STAGES;
  uint64_t* accfull = empty + KX_STAGES;  // [2]
  uint64_t* accempty = accfull + 2;       // [2]
  uint64_t* imgfull = accempty + 2;
  uint64_t* imgfree = imgfull + 1;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort, s_skip;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_abort = 0;
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < KX_STAGES; ++i) {
      mbar_init(smem_u32(&full[i]), 1);
      mbar_init(smem_u32(&empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&accfull[i]), 1);
      mbar_init(smem_u32(&accempty[i]), 4);
    }
    mbar_init(smem_u32(imgfull), 2);  // the bulk copies' arrival + the builder's mu' rows
    mbar_init(smem_u32(imgfree), 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (s_skip) return;
  if (warp == 1) {
    tmem_alloc(smem_u32(&s_tmem), KX_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  volatile int* abort = &s_abort;

  if (warp == 0) {
    // ------------------------------------------------ TMA: key tiles ------
    if (lane == 0) {
      prefetch_tmap(&kmap);
      uint32_t it = 0;
      bool ok = true;
      Item item;
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        for (int64_t t = item.t0; t < item.t1; t += TILE) {
          const int st = it % KX_STAGES;
          if (it >= (uint32_t)KX_STAGES &&
              !mbar_wait(smem_u32(&empty[st]), ((it / KX_STAGES) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          uint8_t* kt = tiles + st * KX_TILE_BYTES;
          mbar_arrive_expect_tx(smem_u32(&full[st]), KX_TILE_BYTES);
          tma_load_4d(smem_u32(kt), &kmap, 0, (int)t, g, l, smem_u32(&full[st]));
          tma_load_4d(smem_u32(kt + KX_BOX), &kmap, 64, (int)t, g, l, smem_u32(&full[st]));
          ++it;
        }
      }
      // no copy may still be landing when the CTA exits
      for (uint32_t k = (it > (uint32_t)KX_STAGES ? it - KX_STAGES : 0); k < it; ++k)
        mbar_wait(smem_u32(&full[k % KX_STAGES]), (k / KX_STAGES) & 1, ws, nullptr);
    }
  } else if (warp == 2) {
    // ------------------------- the unit's image, once per run ------------
    // single buffer: a run's image is written once the previous run's MMAs
    // have all completed (imgfree)
    uint32_t n = 0;
    bool cont = false;
    Item item;
    for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
      const bool same = cont;
      cont = is.next_same_unit(item);
      if (same) continue;
      if (n >= 1 && !mbar_wait(smem_u32(imgfree), (n - 1) & 1, ws, abort)) break;
      const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
      if (lane == 0) {
        const uint8_t* src = ws.qimg + (((int64_t)item.seq * dm.L + l) * dm.Hkv + g) * (int64_t)C::QIMG_BYTES;
        mbar_arrive_expect_tx(smem_u32(imgfull), 4 * C::RP * 128);
#pragma unroll
        for (int a = 0; a < 2; ++a) {
          const uint8_t* sa = src + a * (256 * C::RP);
          bulk_g2s(smem_u32(img + a * C::ATOM), sa, C::RP * 128, smem_u32(imgfull));
          bulk_g2s(smem_u32(img + a * C::ATOM + C::SEC), sa + C::RP * 128, C::RP * 128, smem_u32(imgfull));
        }
      }
      const int64_t qb = (((int64_t)item.seq * dm.L + l) * dm.Hq + (int64_t)g * G) * D;
      write_mu_rows<G, W>(img, ws.mu + qb, lane);
      if (n == 0)  // the zero rows of section 1 (never rewritten)
        for (int e = lane; e < 2 * C::NB * 8; e += 32) {
          const int a = e / (C::NB * 8), r = (e / 8) % C::NB, cc = e % 8;
          *(uint4*)(img + a * C::ATOM + C::SEC + sw128_off(C::RP + r, cc)) = make_uint4(0u, 0u, 0u, 0u);
        }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(imgfull));
      ++n;
    }
    // no image copy may still be landing when the CTA exits
    if (lane == 0 && n > 0) mbar_wait(smem_u32(imgfull), (n - 1) & 1, ws, nullptr);
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer ----------
    if (lane == 0) {
      uint32_t it = 0, n = 0;  // n: runs started
      bool ok = true, cont = false;
      Item item;
      const uint64_t b0 = smem_desc_sw128(smem_u32(img), 16, 1024);
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        if (!cont) {
          if (!mbar_wait(smem_u32(imgfull), n & 1, ws, abort)) break;
          tc_fence_after();
        }
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int st = it % KX_STAGES, slot = it & 1;
          if (!mbar_wait(smem_u32(&full[st]), (it / KX_STAGES) & 1, ws, abort) ||
              (it >= 2 && !mbar_wait(smem_u32(&accempty[slot]), ((it >> 1) & 1) ^ 1, ws, abort))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t a0 = smem_desc_sw128(smem_u32(tiles + st * KX_TILE_BYTES), 16, 1024);
          const uint32_t dacc = tmem + slot * C::ACC;
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {  // descriptors advance by (byte offset >> 4)
            const uint64_t ad = a0 + (uint64_t)((((k >> 2) * KX_BOX) + (k & 3) * 32) >> 4);
            const uint64_t bh = b0 + (uint64_t)((((k >> 2) * C::ATOM) + (k & 3) * 32) >> 4);
            umma_f16_ss(dacc, ad, bh, C::IDESC, k > 0 ? 1u : 0u);
            umma_f16_ss(dacc, ad, bh + (uint64_t)(C::SEC >> 4), C::IDESC, 1u);
          }
          umma_commit(smem_u32(&accfull[slot]));
          umma_commit(smem_u32(&empty[st]));
        }
        if (!ok) break;
        cont = is.next_same_unit(item);
        if (!cont) {
          umma_commit(smem_u32(imgfree));
          ++n;
        }
      }
      // every MMA issued here completes before the CTA tears down tensor memory
      if (it > 0) mbar_wait(smem_u32(&accfull[(it - 1) & 1]), ((it - 1) >> 1) & 1, ws, nullptr);
    }
  } else if (warp >= KX_READ0) {
    // ------------------------------------------------ readout -------------
    const int quarter = warp & 3;
    const int rw = warp - KX_READ0;
    const int y = quarter * 32 + lane;  // token row of the tile (tensor-memory lane)
    const uint32_t lanes = (uint32_t)(quarter * 32) << 16;
    const float invw = 1.f / (float)(dm.cov_unbiased ? dm.window - 1 : dm.window);
    uint32_t it = 0;
    bool bad = false, cont = false;
    float run_m[G], run_s[G];
    Item item;
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
        const int slot = it & 1;
        if (!mbar_wait(smem_u32(&accfull[slot]), (it >> 1) & 1, ws, abort)) break;  // abort: see below
        tc_fence_after();
        const uint32_t ta = tmem + slot * C::ACC + lanes;
        float kap[G];
#pragma unroll
        for (int h = 0; h < G; ++h) kap[h] = 0.f;
#pragma unroll
        for (int b = 0; b < C::RP / 32; b += 2) {
          uint32_t xa[32], xb[32];
          if (b + 1 < C::RP / 32) {
            tmem_ld32x2(ta + b * 32, ta + (b + 1) * 32, xa, xb);
          } else {
            tmem_ld32(ta + b * 32, (float*)xa);
          }
#pragma unroll
          for (int jj = 0; jj < 32; ++jj) {
            const int r = b * 32 + jj;
            if (r < G * W) {
              const float c = __uint_as_float(xa[jj]);
              kap[r / W] = fmaf(c, c, kap[r / W]);
            }
          }
          if (b + 1 < C::RP / 32) {
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
              const int r = (b + 1) * 32 + jj;
              if (r < G * W) {
                const float c = __uint_as_float(xb[jj]);
                kap[r / W] = fmaf(c, c, kap[r / W]);
              }
            }
          }
        }
        float dv[C::NB];
        if constexpr (C::NB == 16) tmem_ld16(ta + C::RP, dv);
        else tmem_ld32(ta + C::RP, dv);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&accempty[slot]));
        const int64_t tok = t + y;
        if (tok < item.t1) {
          float row[2 * G];
#pragma unroll
          for (int h = 0; h < G; ++h) {
            const float lg = dv[h] + dv[G + h] + dv[2 * G + h];
            bad |= !isfinite(lg);
            // branch-free online update: one of the two exponentials is exp(0);
            // both arguments are <= 0 (fast exponential, as in the K pass)
            const float mn = fmaxf(run_m[h], lg);
            run_s[h] = run_s[h] * __expf(run_m[h] - mn) + __expf(lg - mn);
            run_m[h] = mn;
            row[h] = lg;
            row[G + h] = kap[h] * invw;
            bad |= !isfinite(row[G + h]);
          }
          float* dst = lkp + tok * (2 * G);
          store_floats<2 * G, LkAlign<G>::ROW>(dst, row);
        }
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
    if (bad) flag(ws, ST_NONFINITE);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, KX_TMEM_COLS);
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
static cudaError_t launch_kpf(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int grid, cudaStream_t st) {
  using C = KxCfg<G, W>;
  static_assert(C::SMEM <= 232448, "shared memory budget");
  cudaError_t e =
      cudaFuncSetAttribute(kpass_full_bf16_kernel<G, W>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)C::SMEM);
  if (e != cudaSuccess) return e;
  JACAP_TRY(launch_pdl(dm.pdl != 0, kpass_full_bf16_kernel<G, W>, grid, KX_THREADS, C::SMEM, st, kmap, dm, ws));
  return cudaGetLastError();
}

template <int G>
static cudaError_t launch_kpf_g(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int grid, cudaStream_t st) {
  switch (dm.window) {
    case 8: if constexpr (kfull_rows_padded(G, 8) > 0) return launch_kpf<G, 8>(kmap, dm, ws, grid, st); break;
    case 16: if constexpr (kfull_rows_padded(G, 16) > 0) return launch_kpf<G, 16>(kmap, dm, ws, grid, st); break;
    case 32: if constexpr (kfull_rows_padded(G, 32) > 0) return launch_kpf<G, 32>(kmap, dm, ws, grid, st); break;
    case 64: if constexpr (kfull_rows_padded(G, 64) > 0) return launch_kpf<G, 64>(kmap, dm, ws, grid, st); break;
    default: break;
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_kpass_full(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int grid, cudaStream_t st) {
  switch (dm.G) {
    case 1: return launch_kpf_g<1>(kmap, dm, ws, grid, st);
    case 2: return launch_kpf_g<2>(kmap, dm, ws, grid, st);
    case 3: return launch_kpf_g<3>(kmap, dm, ws, grid, st);
    case 4: return launch_kpf_g<4>(kmap, dm, ws, grid, st);
    case 5: return launch_kpf_g<5>(kmap, dm, ws, grid, st);
    case 6: return launch_kpf_g<6>(kmap, dm, ws, grid, st);
    case 7: return launch_kpf_g<7>(kmap, dm, ws, grid, st);
    case 8: return launch_kpf_g<8>(kmap, dm, ws, grid, st);
    default: return cudaErrorInvalidValue;
  }
}

// The tensor-core kernel reads the image that the query statistics wrote
// exactly when dm.kf_rp is set (bf16 cache and a supported shape).
bool kfull_uses_tensor_cores(const Dims& dm, int dtype) { return dtype == 1 && dm.kf_rp > 0; }

cudaError_t launch_kfull(const CUtensorMap& kmap, const Dims& dm, const Ws& ws, int dtype, const void* k, int grid,
                         cudaStream_t st) {
  (void)kmap;
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
