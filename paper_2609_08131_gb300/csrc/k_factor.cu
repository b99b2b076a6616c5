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
// d_j = A_jj and the right block holds X = Lt^{-1}, where A = Lt U with Lt
// unit lower triangular and U = Diag(d) Lt^T, so L = Lt Diag(d)^{1/2} and
// L^{-1} = Diag(d)^{-1/2} X. Both blocks live in registers: thread (ty, tx)
// of the 16 x 32 thread grid owns rows ty + 16a and columns tx + 32b of A and
// X; each step broadcasts column j of A (equal to row j by symmetry of every
// Schur complement) and row j of X through double-buffered shared memory, so
// a step costs one barrier and at most 64 fused multiply-adds per thread.
//
// L^{-1} is written twice: as float32 (used by the float32 score pass and
// exposed for tests) and as a bf16 hi/lo pair laid out exactly as the
// shared-memory B operand of the tensor-core score pass (K-major, 128-byte
// swizzle): rows n < 128 hold hi(L^{-1}[n, :]), rows n >= 128 hold
// lo(L^{-1}[n-128, :]) = L^{-1} - hi rounded again, so hi + lo carries ~16
// significant bits.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int FA_THREADS = 512;
constexpr int FA_LD = D + 1;
constexpr size_t factor_smem_bytes() { return (size_t)D * FA_LD * sizeof(float); }

__global__ void __launch_bounds__(FA_THREADS, 1) factor_kernel(Dims dm, Ws ws) {
  extern __shared__ float Ms[];  // [D][FA_LD]: L^{-1} staged for the bf16 image
  __shared__ float colA[2][D], rowX[2][D], piv[D];
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
  const int c0 = ws.plan[1 + s], c1 = ws.plan[2 + s];
  const int ty = tid >> 5, tx = tid & 31;

  // A = I + sum of partial Grams (chunk order); X = I
  float ar[8][4], xr[8][4];
  {
    const float* gp = ws.gpart + ((int64_t)plane * dm.c_cap) * D * D;
    float* gout = ws.gram + (int64_t)u * D * D;
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) ar[a][b] = 0.f;
    for (int ch = c0; ch < c1; ++ch) {  // 32 independent loads in flight per chunk
      // partial layout: (m, n) at ((n / 32) D + m) 32 + n % 32, so a warp
      // (fixed row, 32 consecutive columns) reads 128 contiguous bytes
      const float* src = gp + (int64_t)ch * D * D;
#pragma unroll
      for (int a = 0; a < 8; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) ar[a][b] += src[(b * D + ty + 16 * a) * 32 + tx];
    }
#pragma unroll
    for (int a = 0; a < 8; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const int i = ty + 16 * a, c = tx + 32 * b;
        gout[i * D + c] = ar[a][b];
        ar[a][b] += (i == c ? 1.f : 0.f);
        xr[a][b] = i == c ? 1.f : 0.f;
      }
  }

  // forward elimination, step j = 32 jb + 16 jh + jj (jb, jh unrolled so the
  // register indices of the pivot column and row are compile-time constants)
#pragma unroll
  for (int jb = 0; jb < 4; ++jb) {
#pragma unroll
    for (int jh = 0; jh < 2; ++jh) {
#pragma unroll 1
      for (int jj = 0; jj < 16; ++jj) {
        const int j = 32 * jb + 16 * jh + jj;
        const int buf = j & 1;
        if (tx == (j & 31)) {  // owners of column j of A (register column jb)
#pragma unroll
          for (int a = 0; a < 8; ++a) colA[buf][ty + 16 * a] = ar[a][jb];
          if (ty == (j & 15)) piv[j] = ar[2 * jb + jh][jb];
        }
        if (ty == (j & 15)) {  // owners of row j of X (register row 2 jb + jh)
#pragma unroll
          for (int b = 0; b < 4; ++b) rowX[buf][tx + 32 * b] = xr[2 * jb + jh][b];
        }
        __syncthreads();
        const float inv_p = 1.f / colA[buf][j];
        float ck[4], rx[4];
#pragma unroll
        for (int b = 0; b < 4; ++b) {
          ck[b] = colA[buf][tx + 32 * b];
          rx[b] = rowX[buf][tx + 32 * b];
        }
#pragma unroll
        for (int a = 0; a < 8; ++a) {
          const int i = ty + 16 * a;
          if (i > j) {
            const float m = colA[buf][i] * inv_p;
#pragma unroll
            for (int b = 0; b < 4; ++b) {
              const int c = tx + 32 * b;
              if (c > j) {
                if (c <= i) ar[a][b] = fmaf(-m, ck[b], ar[a][b]);
              } else {
                xr[a][b] = fmaf(-m, rx[b], xr[a][b]);
              }
            }
          }
        }
      }
    }
  }
  __syncthreads();

  // L^{-1} = Diag(d)^{-1/2} X
  float* mout = ws.minv + (int64_t)u * D * D;
#pragma unroll
  for (int a = 0; a < 8; ++a) {
    const int i = ty + 16 * a;
    const float d = piv[i];
    if (!(d > 0.f) || !isfinite(d)) s_bad = 1;
    const float sc = 1.f / sqrtf(fmaxf(d, 1e-30f));
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int c = tx + 32 * b;
      const float x = xr[a][b] * sc;
      if (!isfinite(x)) s_bad = 1;
      mout[i * D + c] = x;
      Ms[i * FA_LD + c] = x;
    }
  }
  __syncthreads();
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

cudaError_t launch_factor(const Dims& dm, const Ws& ws, cudaStream_t st) {
  constexpr size_t smem = factor_smem_bytes();
  cudaError_t e = cudaFuncSetAttribute(factor_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int units = dm.L * dm.Hkv * dm.S;
  factor_kernel<<<units, FA_THREADS, smem, st>>>(dm, ws);
  return cudaGetLastError();
}

}  // namespace jacap
