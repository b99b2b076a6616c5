// k_score.cu - Jacap scores r_i = w_i v_i^T A^{-1} v_i = w_i ||L^{-1} v_i||^2 (Eq. 10).
//
// bf16 caches: the tensor cores form Y = V (L^{-1})^T for a 128-token tile:
// hi(L^{-1}) and lo(L^{-1}) (K-major, from a 64 KB shared-memory image written
// by the factor kernel) accumulate into the same 128 fp32 columns, so
// y = V (hi + lo)^T. L^{-1} is lower triangular, so output columns 0-63 need
// only channels 0-63: the first four K-steps are N = 128 MMAs, the last four
// N = 64 MMAs into columns 64-127. The image's zero quarter (rows 0-63 of
// channels 64-127) is not copied into shared memory, which leaves room for a
// fourth V stage. V comes straight from the TMA-staged tile; a warp of its
// own loads the images, so the V ring never waits behind an image slot.
// Each epilogue thread owns one token (one TMEM lane) and reduces
// ||y||^2 = sum_j D[j]^2 in fp32, then multiplies by w_i. The tensor-memory accumulator
// is double-buffered so the epilogue of tile i overlaps the MMAs of tile i+1,
// and so is the L^{-1} image: it is loaded once per run of consecutive items
// of one unit, and the next unit's image streams in while the current run's
// tiles go through.
// float32 caches: SIMT forward products with L^{-1} held in shared memory.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int SC_THREADS = 224;  // warp 0: V tiles (TMA), warp 1: MMA, warps 2-5: epilogue, warp 6: images
template <bool DENSE> __host__ __device__ constexpr int sc_stages() { return DENSE ? 3 : 4; }  // V tiles in flight
template <bool DENSE> __host__ __device__ constexpr int sc_imgs() { return 2; }  // L^{-1} image buffers
constexpr int SC_BOX = 16384;
constexpr int SC_TILE_BYTES = 2 * SC_BOX;
constexpr int SC_M_BYTES = 65536;
constexpr uint32_t SC_TMEM_COLS = 256;  // two 128-column accumulators
// M = 128 tokens, N = 128 or 64 rows of the L^{-1} image, both operands K-major.
constexpr uint32_t SC_IDESC128 = idesc_bf16_f32(128, 128, 0, 0);
constexpr uint32_t SC_IDESC64 = idesc_bf16_f32(128, 64, 0, 0);

// the lower-triangular image without its zero quarter: channel atom 0 whole
// (32 KB), then rows 64-127 of atom 1 for hi (8 KB) and for lo (8 KB)
constexpr int SC_MT_BYTES = 49152;
template <bool DENSE> __host__ __device__ constexpr int sc_img_bytes() { return DENSE ? SC_M_BYTES : SC_MT_BYTES; }
template <bool DENSE>
constexpr size_t score_bf16_smem_bytes() {
  return 1024 + sc_imgs<DENSE>() * sc_img_bytes<DENSE>() + sc_stages<DENSE>() * SC_TILE_BYTES + 256;
}

// DENSE: the score matrix is a full 128 x 128 (output directions) rather than
// the lower-triangular L^{-1}, so no K-step may be narrowed.
template <bool DENSE>
__global__ void __launch_bounds__(SC_THREADS, 1)
    score_bf16_kernel(const __grid_constant__ CUtensorMap vmap, Dims dm, Ws ws, const int32_t* __restrict__ cu,
                      float* __restrict__ scores) {
  pdl_wait();
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
      mbar_init(smem_u32(&accempty[i]), 4);
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
    tmem_alloc(smem_u32(&s_tmem), SC_TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  volatile int* abort = &s_abort;

  if (warp == 0) {
    if (lane == 0) {
      prefetch_tmap(&vmap);
      uint32_t it = 0;
      bool ok = true;
      Item item;
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
        for (int64_t t = item.t0; t < item.t1; t += TILE) {
          const int st = it % SC_STAGES;
          if (it >= (uint32_t)SC_STAGES &&
              !mbar_wait(smem_u32(&vempty[st]), ((it / SC_STAGES) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          uint8_t* vt = stages + st * SC_TILE_BYTES;
          mbar_arrive_expect_tx(smem_u32(&vfull[st]), SC_TILE_BYTES);
          tma_load_4d(smem_u32(vt), &vmap, 0, (int)t, g, l, smem_u32(&vfull[st]));
          tma_load_4d(smem_u32(vt + SC_BOX), &vmap, 64, (int)t, g, l, smem_u32(&vfull[st]));
          ++it;
        }
      }
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
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
        const bool same = cont;
        cont = is.next_same_unit(item);
        if (same) continue;
        const int64_t u = (int64_t)item.plane * dm.S + item.seq;
        const int mp = nrun % SC_IMGS;
        if (nrun >= SC_IMGS && !mbar_wait(smem_u32(&mempty[mp]), ((nrun / SC_IMGS) & 1) ^ 1, ws, abort)) break;
        mbar_arrive_expect_tx(smem_u32(&mfull[mp]), IMG);
        const uint8_t* src = ws.minv_img + u * SC_M_BYTES;
        uint8_t* dst = mimg + mp * IMG;
        if (DENSE) {
          bulk_g2s(smem_u32(dst), src, SC_M_BYTES, smem_u32(&mfull[mp]));
        } else {
          bulk_g2s(smem_u32(dst), src, 32768, smem_u32(&mfull[mp]));
          bulk_g2s(smem_u32(dst + 32768), src + 32768 + 8192, 8192, smem_u32(&mfull[mp]));
          bulk_g2s(smem_u32(dst + 40960), src + 32768 + 24576, 8192, smem_u32(&mfull[mp]));
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
      for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); ok && is.next(item);) {
        if (!cont) {
          mp = nrun % SC_IMGS;
          if (!mbar_wait(smem_u32(&mfull[mp]), (nrun / SC_IMGS) & 1, ws, abort)) break;
          tc_fence_after();
        }
        const uint32_t ma = smem_u32(mimg + mp * IMG);
        for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
          const int st = it % SC_STAGES;
          const int ab = it & 1;
          if (it >= 2 && !mbar_wait(smem_u32(&accempty[ab]), ((it >> 1) & 1) ^ 1, ws, abort)) {
            ok = false;
            break;
          }
          if (!mbar_wait(smem_u32(&vfull[st]), (it / SC_STAGES) & 1, ws, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // descriptors advance by (byte offset >> 4); image rows: hi at row n,
          // lo at row 128 + n (16 KB further) of each 32 KB channel atom
          const uint64_t a0 = smem_desc_sw128(smem_u32(stages + st * SC_TILE_BYTES), 16, 1024);
          const uint64_t b0 = smem_desc_sw128(ma, 16, 1024);
          const uint32_t dacc = tmem + ab * 128;
#pragma unroll
          for (int k = 0; k < D / 16; ++k) {  // 16 channels per K-step
            const uint64_t ad = a0 + (uint64_t)((((k >> 2) * SC_BOX) + (k & 3) * 32) >> 4);
            const uint64_t bk = b0 + (uint64_t)((((k >> 2) * 32768) + (k & 3) * 32) >> 4);
            if (k < 4 || DENSE) {  // channels 0-63 (or a full matrix): all 128 output columns
              umma_f16_ss(dacc, ad, bk, SC_IDESC128, k > 0 ? 1u : 0u);
              umma_f16_ss(dacc, ad, bk + (16384 >> 4), SC_IDESC128, 1u);
            } else {      // channels 64-127: only columns (rows of L^{-1}) 64-127 are nonzero
              const uint64_t bt = b0 + (uint64_t)((32768 + (k & 3) * 32) >> 4);
              umma_f16_ss(dacc + 64, ad, bt, SC_IDESC64, 1u);
              umma_f16_ss(dacc + 64, ad, bt + (8192 >> 4), SC_IDESC64, 1u);
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
    }
  } else if (warp < 6) {
    const int quarter = warp & 3;
    const int y = quarter * 32 + lane;  // token row of the tile == TMEM lane
    uint32_t it = 0;
    bool bad = false;
    Item item;
    for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
      for (int64_t t = item.t0; t < item.t1; t += TILE, ++it) {
        const int ab = it & 1;
        const int64_t tok = t + y;
        const int64_t o = (int64_t)item.plane * dm.Ntot + tok;
        const float wt = tok < item.t1 ? ws.w[o] : 0.f;  // issued before the wait: hides its latency
        if (!mbar_wait(smem_u32(&accfull[ab]), (it >> 1) & 1, ws, abort)) goto epi_done;
        tc_fence_after();
        const uint32_t trow = tmem + ab * 128 + ((uint32_t)(quarter * 32) << 16);
        float ssq = 0.f;
#pragma unroll 1
        for (int cb = 0; cb < 4; ++cb) {
          float a[32];
          tmem_ld32(trow + cb * 32, a);
#pragma unroll
          for (int j = 0; j < 32; ++j) ssq = fmaf(a[j], a[j], ssq);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&accempty[ab]));
        if (tok < item.t1) {
          const float sc = wt * ssq;
          scores[o] = sc;
          bad |= !isfinite(sc);
        }
      }
    }
  epi_done:
    if (bad) flag(ws, ST_NONFINITE);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, SC_TMEM_COLS);
  }
}

// ------------------------------------------------------------ SIMT fp32 ---
// Two threads per token (lanes 2 t and 2 t + 1): thread `half` forms the
// output rows r of the quads r / 4 = half, half + 2, ... (the two halves of
// the triangle get about the same work), four rows at once so their
// multiply-add chains interleave, and the pair adds its squared norms.
// L^{-1} is stored with zeros above the diagonal, so a quad may run its
// columns up to its last row.
constexpr int SF_THREADS = 2 * TILE;
constexpr int SF_LD = D + 1;
constexpr size_t score_f32_smem_bytes() { return (size_t)(D * D + TILE * SF_LD) * sizeof(float); }

__global__ void __launch_bounds__(SF_THREADS)
    score_f32_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu, const float* __restrict__ v,
                     float* __restrict__ scores) {
  pdl_wait();
  extern __shared__ float ssm[];
  float* Mi = ssm;               // [D][D] L^{-1}
  float* vt = ssm + D * D;       // [TILE][SF_LD]
  __shared__ int s_skip;
  const int tid = threadIdx.x;
  if (tid == 0) s_skip = status_failed(ws) ? 1 : 0;
  __syncthreads();
  if (s_skip) return;
  const int tk = tid >> 1, half = tid & 1;
  bool bad = false;
  int64_t loaded = -1;
  Item item;
  for (ItemStream is(dm, ws, blockIdx.x, gridDim.x); is.next(item);) {
    const int l = item.plane / dm.Hkv, g = item.plane % dm.Hkv;
    const int64_t u = (int64_t)item.plane * dm.S + item.seq;
    const float* vbase = v + (int64_t)l * dm.kv_sl + (int64_t)g * dm.kv_sh;
    __syncthreads();
    if (u != loaded) {
      const float* src = ws.minv + u * D * D;
      for (int e = tid * 4; e < D * D; e += SF_THREADS * 4) *(float4*)(Mi + e) = *(const float4*)(src + e);
      loaded = u;
    }
    for (int64_t t = item.t0; t < item.t1; t += TILE) {
      __syncthreads();
      for (int e = tid; e < TILE * (D / 4); e += SF_THREADS) {
        const int r = e / (D / 4), c4 = (e % (D / 4)) * 4;
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (t + r < item.t1) x = *(const float4*)(vbase + (t + r) * dm.kv_st + c4);
        vt[r * SF_LD + c4] = x.x; vt[r * SF_LD + c4 + 1] = x.y;
        vt[r * SF_LD + c4 + 2] = x.z; vt[r * SF_LD + c4 + 3] = x.w;
      }
      __syncthreads();
      const float* vr = vt + tk * SF_LD;
      float ssq = 0.f;
      for (int r0 = 4 * half; r0 < D; r0 += 8) {
        const float* m0 = Mi + r0 * D;
        // a full matrix with output directions
        const int cend = dm.dense_minv ? D : r0 + 4;
        float y0 = 0.f, y1 = 0.f, y2 = 0.f, y3 = 0.f;
        for (int c = 0; c < cend; ++c) {
          const float x = vr[c];
          y0 = fmaf(m0[c], x, y0);
          y1 = fmaf(m0[D + c], x, y1);
          y2 = fmaf(m0[2 * D + c], x, y2);
          y3 = fmaf(m0[3 * D + c], x, y3);
        }
        ssq = fmaf(y0, y0, fmaf(y1, y1, fmaf(y2, y2, fmaf(y3, y3, ssq))));
      }
      ssq += __shfl_xor_sync(0xffffffffu, ssq, 1);
      const int64_t tok = t + tk;
      if (half == 0 && tok < item.t1) {
        const int64_t o = (int64_t)item.plane * dm.Ntot + tok;
        const float sc = ws.w[o] * ssq;
        scores[o] = sc;
        bad |= !isfinite(sc);
      }
    }
  }
  if (bad) flag(ws, ST_NONFINITE);
}

cudaError_t launch_score(const CUtensorMap& vmap, const Dims& dm, const Ws& ws, int dtype, const void* v,
                         const int32_t* cu, float* scores, int grid, cudaStream_t st) {
  if (dtype == 1) {
    const size_t smem = dm.dense_minv ? score_bf16_smem_bytes<true>() : score_bf16_smem_bytes<false>();
    static_assert(score_bf16_smem_bytes<true>() <= 232448 && score_bf16_smem_bytes<false>() <= 232448, "smem");
    auto kern = dm.dense_minv ? score_bf16_kernel<true> : score_bf16_kernel<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    JACAP_TRY(launch_pdl(dm.pdl != 0, kern, grid, SC_THREADS, smem, st, vmap, dm, ws, cu, scores));
  } else {
    constexpr size_t smem = score_f32_smem_bytes();
    cudaError_t e = cudaFuncSetAttribute(score_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    JACAP_TRY(launch_pdl(dm.pdl != 0, score_f32_kernel, grid, SF_THREADS, smem, st, dm, ws, cu, (const float*)v,
                         scores));
  }
  return cudaGetLastError();
}

}  // namespace jacap
