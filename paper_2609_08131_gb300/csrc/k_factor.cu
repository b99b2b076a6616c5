// k_factor.cu - capacity matrix and the inverse of its Cholesky factor, one
// CTA per unit.
//
//  G        = sum over the unit's chunks of the partial Grams  (Eq. 9 without I)
//  A        = I + G                                           (Eq. 9, Sigma_noise = I)
//  L^{-1}   where A = L L^T.
//
// Since v^T A^{-1} v = ||L^{-1} v||^2, the score pass needs only L^{-1}
// (Eq. 10). It is obtained by Gaussian forward elimination of [A | I] without
// pivoting (safe: A is symmetric positive definite): after step j the pivot
// p_j = A_jj and the right block holds X = Lt^{-1}, where A = Lt U with Lt
// unit lower triangular and U = Diag(p) Lt^T, so L = Lt Diag(p)^{1/2} and
// L^{-1} = Diag(p)^{-1/2} X.
//
// Both blocks share one 128 x 128 register array Z: column c holds A until
// step c eliminates it, and afterwards Y_c = -p_c X_{., c}. In that scaling
// the eliminated value A_ic (= m_i p_c with m_i = A_ic / p_c) already equals
// Y_ic, so step j updates every active row i > j by the same fused
// multiply-add Z_i. -= m_i r with r_c = A_cj (c > j, lower triangle of A by
// symmetry), r_j = 0 and r_c = Z_jc (c < j, row j of Y): one barrier and at
// most 64 multiply-adds per thread. At the end X_ic = -Y_ic / p_c. Thread
// (ty, tx) of the 8 x 32 grid owns rows ty + 8 a and columns 4 tx .. 4 tx + 3;
// with 256 threads two units share an SM, so their barrier latencies overlap.
// The multipliers use 1/p_j from the approximate hardware reciprocal refined by
// one Newton-Raphson step (x <- x (2 - p x)), which is accurate to about one ulp.
//
// With output directions u = W v (Sec. 3.1) the capacity matrix I + sum w u u^T
// lives in the output space; with a 128 x 128 factor F of W^T W (F^T F = W^T W)
// it reduces exactly to M = I + F G F^T, and u^T A^{-1} u = ||L_M^{-1} F v||^2.
// That variant forms F G F^T from shared-memory copies of G and F (three
// SIMT float32 products of 128 x 128 matrices), factors M as below and writes
// T = L_M^{-1} F in place of L^{-1}.
//
// L^{-1} is written twice: as float32 (used by the float32 score pass and
// exposed for tests) and as a bf16 hi/lo pair laid out exactly as the
// shared-memory B operand of the tensor-core score pass (K-major, 128-byte
// swizzle, two 64-channel atoms of 256 rows): hi(L^{-1}[n, :]) at row
// 32 (n / 16) + n % 16 and lo(L^{-1}[n, :]) = L^{-1} - hi rounded again 16
// rows further (hi and lo interleaved by 16-row blocks, so the rows a K-step
// of the triangular product needs are contiguous), so hi + lo carries ~16
// significant bits. The output-direction variant (T = L_M^{-1} F, a full
// matrix) keeps hi in rows 0-127 and lo in rows 128-255.
#include "jacap_dev.cuh"
#include "jacap_internal.h"
#include "k_factor_body.cuh"

namespace jacap {

constexpr int FA_LD = D + 1;
// PROJ: two padded 128 x 128 float32 matrices (R0: G, then F G, then L^{-1},
// then the image staging; R1: F); otherwise the staging matrix only.
template <bool PROJ>
constexpr size_t factor_smem_bytes() { return (size_t)(PROJ ? 2 : 1) * D * FA_LD * sizeof(float); }

template <bool PROJ>
__global__ void __launch_bounds__(FA_THREADS, PROJ ? 1 : 2)
    factor_kernel(Dims dm, Ws ws, const float* __restrict__ out_factor) {
  pdl_wait();
  extern __shared__ float Ms[];  // [D][FA_LD]: L^{-1} staged for the bf16 image (PROJ: R0, then R1)
  __shared__ __align__(16) float colA[2][D];
  __shared__ __align__(16) float rowY[2][D];
  __shared__ float piv[D];
  __shared__ int s_skip, s_bad;
  const int tid = threadIdx.x;
  if (tid == 0) {
    s_skip = status_failed(ws) ? 1 : 0;
    s_bad = 0;
  }
  __syncthreads();
  if (s_skip) return;
  const int u = blockIdx.x;
  const int plane = u / dm.S, s = u % dm.S;
  const int ch0 = ws.plan[1 + s], ch1 = ws.plan[2 + s];
  const int ty = tid >> 5, tx = tid & 31;
  const int c0 = 4 * tx;

  // A = I + sum of partial Grams (chunk order)
  float2 z[FA_ROWS][2];  // columns (c0, c0+1) and (c0+2, c0+3) as packed pairs
  {
    const float* gp = ws.gpart + ((int64_t)plane * dm.c_cap) * D * D;
    float* gout = ws.gram + (int64_t)u * D * D;
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a) z[a][0] = z[a][1] = make_float2(0.f, 0.f);
    const int32_t* pf = ws.pflag + (int64_t)plane * dm.c_cap;
    for (int ch = ch0; ch < ch1; ++ch) {  // 16 independent 16-byte loads in flight per chunk
      if (!pf[ch]) continue;  // no partial at this chunk (it continued a run)
      // partial layout: (m, n) at ((n / 32) D + m) 32 + n % 32; only the
      // lower 32 x 32 blocks are stored (rows ty + 8 a lie in block a / 4)
      const float* src = gp + (int64_t)ch * D * D + (c0 >> 5) * D * 32 + (c0 & 31);
#pragma unroll
      for (int a = 0; a < FA_ROWS; ++a) {
        if (a / 4 < (c0 >> 5)) continue;
        const float4 v = *(const float4*)(src + (ty + 8 * a) * 32);
        z[a][0].x += v.x;
        z[a][0].y += v.y;
        z[a][1].x += v.z;
        z[a][1].y += v.w;
      }
    }
    // the upper blocks by symmetry, through the staging matrix
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a) {
      const int i = ty + 8 * a;
      if (a / 4 < (c0 >> 5)) continue;
      Ms[i * FA_LD + c0] = z[a][0].x;
      Ms[i * FA_LD + c0 + 1] = z[a][0].y;
      Ms[i * FA_LD + c0 + 2] = z[a][1].x;
      Ms[i * FA_LD + c0 + 3] = z[a][1].y;
    }
    __syncthreads();
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a) {
      const int i = ty + 8 * a;
      if (a / 4 < (c0 >> 5))
        z[a][0] = make_float2(Ms[c0 * FA_LD + i], Ms[(c0 + 1) * FA_LD + i]),
        z[a][1] = make_float2(Ms[(c0 + 2) * FA_LD + i], Ms[(c0 + 3) * FA_LD + i]);
      *(float4*)(gout + i * D + c0) = make_float4(z[a][0].x, z[a][0].y, z[a][1].x, z[a][1].y);
    }
    __syncthreads();
  }
  if constexpr (PROJ) {
    // M = F G F^T: G and F to shared memory (stride FA_LD), then two products
    // with thread (ty, tx) computing rows ty + 8 a, columns tx + 32 b
    float* R0 = Ms;
    float* R1 = Ms + D * FA_LD;
    const float* F = out_factor + (int64_t)plane * D * D;
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a) {
      const int i = ty + 8 * a;
      R0[i * FA_LD + c0] = z[a][0].x;
      R0[i * FA_LD + c0 + 1] = z[a][0].y;
      R0[i * FA_LD + c0 + 2] = z[a][1].x;
      R0[i * FA_LD + c0 + 3] = z[a][1].y;
    }
    for (int e = tid; e < D * D / 4; e += FA_THREADS) {
      const float4 f = ((const float4*)F)[e];
      const int r = e / (D / 4), c = (e % (D / 4)) * 4;
      R1[r * FA_LD + c] = f.x;
      R1[r * FA_LD + c + 1] = f.y;
      R1[r * FA_LD + c + 2] = f.z;
      R1[r * FA_LD + c + 3] = f.w;
    }
    __syncthreads();
    float acc[FA_ROWS][4];
    // T1 = F G: T1[i][c] = sum_m F[i][m] G[m][c]
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
#pragma unroll 2
    for (int m = 0; m < D; ++m) {
      float g[4];
#pragma unroll
      for (int b = 0; b < 4; ++b) g[b] = R0[m * FA_LD + tx + 32 * b];
#pragma unroll
      for (int a = 0; a < FA_ROWS; ++a) {
        const float f = R1[(ty + 8 * a) * FA_LD + m];
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(f, g[b], acc[a][b]);
      }
    }
    __syncthreads();
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) R0[(ty + 8 * a) * FA_LD + tx + 32 * b] = acc[a][b];
    __syncthreads();
    // M = T1 F^T: M[i][c] = sum_m T1[i][m] F[c][m]
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
#pragma unroll 2
    for (int m = 0; m < D; ++m) {
      float f[4];
#pragma unroll
      for (int b = 0; b < 4; ++b) f[b] = R1[(tx + 32 * b) * FA_LD + m];
#pragma unroll
      for (int a = 0; a < FA_ROWS; ++a) {
        const float t = R0[(ty + 8 * a) * FA_LD + m];
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(t, f[b], acc[a][b]);
      }
    }
    __syncthreads();
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) R0[(ty + 8 * a) * FA_LD + tx + 32 * b] = acc[a][b];
    __syncthreads();
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a) {
      const int i = ty + 8 * a;
      z[a][0] = make_float2(R0[i * FA_LD + c0], R0[i * FA_LD + c0 + 1]);
      z[a][1] = make_float2(R0[i * FA_LD + c0 + 2], R0[i * FA_LD + c0 + 3]);
    }
    __syncthreads();
  }
  {
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a) {
      const int i = ty + 8 * a;
      z[a][0].x += (i == c0 ? 1.f : 0.f);
      z[a][0].y += (i == c0 + 1 ? 1.f : 0.f);
      z[a][1].x += (i == c0 + 2 ? 1.f : 0.f);
      z[a][1].y += (i == c0 + 3 ? 1.f : 0.f);
    }
  }

  // forward elimination, step j = 8 jh + jl (jl unrolled so the register
  // column of the pivot column is a compile-time constant)
#pragma unroll 1
  for (int jh = 0; jh < 16; ++jh) {
#pragma unroll
    for (int jl = 0; jl < 8; ++jl) {
      const int j = 8 * jh + jl;
      const int buf = j & 1;
      if (tx == (j >> 2)) {  // owners of column j: rows ty + 8 a, register column j % 4 = jl % 4
#pragma unroll
        for (int a = 0; a < FA_ROWS; ++a) {
          const float2 zp = z[a][(jl & 3) >> 1];
          colA[buf][ty + 8 * a] = (jl & 1) ? zp.y : zp.x;
        }
      }
      if (ty == jl) {  // owners of row j (register row jh)
        float2 r01 = make_float2(0.f, 0.f), r23 = r01;
#pragma unroll
        for (int a = 0; a < FA_ROWS; ++a)
          if (a == jh) {
            r01 = z[a][0];
            r23 = z[a][1];
          }
        *(float4*)&rowY[buf][c0] = make_float4(r01.x, r01.y, r23.x, r23.y);
      }
      __syncthreads();
      const float pj = colA[buf][j];
      if (tid == 0) piv[j] = pj;
      const float inv_p = recip_nr(pj);
      const float4 ca = *(const float4*)&colA[buf][c0];
      const float4 ry = *(const float4*)&rowY[buf][c0];
      const float cav[4] = {ca.x, ca.y, ca.z, ca.w}, ryv[4] = {ry.x, ry.y, ry.z, ry.w};
      float r[4];
#pragma unroll
      for (int b = 0; b < 4; ++b) r[b] = c0 + b > j ? cav[b] : (c0 + b == j ? 0.f : ryv[b]);
      const float2 r01 = make_float2(r[0], r[1]), r23 = make_float2(r[2], r[3]);
#pragma unroll
      for (int a = 0; a < FA_ROWS; ++a) {
        if (ty + 8 * a > j) {  // active rows (uniform over the warp)
          const float m = colA[buf][ty + 8 * a] * inv_p;
          const float2 nm = make_float2(-m, -m);
          z[a][0] = __ffma2_rn(nm, r01, z[a][0]);
          z[a][1] = __ffma2_rn(nm, r23, z[a][1]);
        }
      }
    }
  }
  __syncthreads();

  // L^{-1}_ic = X_ic / sqrt(p_i) with X_ic = -Y_ic / p_c (c < i), X_ii = 1
  float* mout = ws.minv + (int64_t)u * D * D;
  float ipc[4];
#pragma unroll
  for (int b = 0; b < 4; ++b) ipc[b] = 1.f / piv[c0 + b];
#pragma unroll
  for (int a = 0; a < FA_ROWS; ++a) {
    const int i = ty + 8 * a;
    const float d = piv[i];
    if (!(d > 0.f) || !isfinite(d)) s_bad = 1;
    const float sc = 1.f / sqrtf(fmaxf(d, 1e-30f));
    const float zv[4] = {z[a][0].x, z[a][0].y, z[a][1].x, z[a][1].y};
    float x[4];
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int c = c0 + b;
      x[b] = c < i ? (-zv[b] * ipc[b]) * sc : (c == i ? sc : 0.f);
      if (!isfinite(x[b])) s_bad = 1;
      Ms[i * FA_LD + c] = x[b];
    }
    if constexpr (!PROJ) *(float4*)(mout + i * D + c0) = make_float4(x[0], x[1], x[2], x[3]);
  }
  __syncthreads();
  if constexpr (PROJ) {
    // T = L_M^{-1} F: T[i][c] = sum_{m <= i} L^{-1}[i][m] F[m][c] (L^{-1} now in R0 = Ms)
    const float* R1 = Ms + D * FA_LD;
    float acc[FA_ROWS][4];
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
#pragma unroll 2
    for (int m = 0; m < D; ++m) {
      float f[4];
#pragma unroll
      for (int b = 0; b < 4; ++b) f[b] = R1[m * FA_LD + tx + 32 * b];
#pragma unroll
      for (int a = 0; a < FA_ROWS; ++a) {
        const float l = Ms[(ty + 8 * a) * FA_LD + m];
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(l, f[b], acc[a][b]);
      }
    }
    __syncthreads();
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int i = ty + 8 * a, c = tx + 32 * b;
        if (!isfinite(acc[a][b])) s_bad = 1;
        Ms[i * FA_LD + c] = acc[a][b];
        mout[i * D + c] = acc[a][b];
      }
    __syncthreads();
  }
  // bf16 hi/lo image: 2 K-atoms (channels 0-63, 64-127) x 256 rows x 128 B
  uint8_t* img = ws.minv_img + (int64_t)u * 65536;
  for (int e = tid; e < 256 * 16; e += FA_THREADS) {
    const int n = e / 16, cc = e % 16;  // row n, 8-channel chunk cc
    const int r = n & 127;
    const bool lo = n >= 128;
    uint32_t wv[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float x0 = Ms[r * FA_LD + cc * 8 + 2 * q];
      const float x1 = Ms[r * FA_LD + cc * 8 + 2 * q + 1];
      const uint32_t h = pack_bf16x2(x0, x1);
      wv[q] = lo ? pack_bf16x2(x0 - bf16lo(h), x1 - bf16hi(h)) : h;
    }
    const uint32_t off = (cc >> 3) * 32768 + sw128_off(n, cc & 7);
    *(uint4*)(img + off) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  }
  __syncthreads();
  if (tid == 0 && s_bad) flag(ws, ST_NONFINITE);
}

__global__ void __launch_bounds__(FB_THREADS, 2) factor_blocked_kernel(Dims dm, Ws ws) {
  pdl_wait();
  factor_blocked_cta<false>(dm, ws, blockIdx.x, gridDim.x);
}

template <bool PROJ>
static cudaError_t launch_factor_t(const Dims& dm, const Ws& ws, const float* out_factor, cudaStream_t st) {
  constexpr size_t smem = factor_smem_bytes<PROJ>();
  cudaError_t e = cudaFuncSetAttribute(factor_kernel<PROJ>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int units = dm.L * dm.Hkv * dm.S;
  JACAP_TRY(launch_pdl(dm.pdl != 0, factor_kernel<PROJ>, units, FA_THREADS, smem, st, dm, ws, out_factor));
  return cudaGetLastError();
}

cudaError_t launch_factor(const Dims& dm, const Ws& ws, const float* out_factor, cudaStream_t st) {
  if (out_factor != nullptr) return launch_factor_t<true>(dm, ws, out_factor, st);
  cudaError_t e = cudaFuncSetAttribute(factor_blocked_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)FB_SMEM);
  if (e != cudaSuccess) return e;
  JACAP_TRY(launch_pdl(dm.pdl != 0, factor_blocked_kernel, dm.L * dm.Hkv * dm.S, FB_THREADS, FB_SMEM, st, dm, ws));
  return cudaGetLastError();
}

}  // namespace jacap
