// k_factor.cu - capacity matrix and its factor, one CTA per unit.
//
//  G        = sum over the unit's chunks of the partial Grams  (Eq. 9 without I)
//  A        = I + G                                           (Eq. 9, Sigma_noise = I)
//  A        = L L^T   (Cholesky, float32, right-looking, in shared memory)
//  L^{-1}   by forward substitution, one column per thread.
//
// Since v^T A^{-1} v = ||L^{-1} v||^2, the score pass needs only L^{-1}
// (Eq. 10). It is written twice: as float32 (used by the float32 score pass
// and exposed for tests) and as a bf16 hi/lo pair laid out exactly as the
// shared-memory B operand of the tensor-core score pass (K-major, 128-byte
// swizzle): rows n < 128 hold hi(L^{-1}[n, :]), rows n >= 128 hold
// lo(L^{-1}[n-128, :]) = L^{-1} - hi rounded again, so hi + lo carries ~16
// significant bits.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int FA_THREADS = 512;
constexpr int FA_LD = D + 1;
constexpr size_t factor_smem_bytes() { return (size_t)2 * D * FA_LD * sizeof(float); }

__global__ void __launch_bounds__(FA_THREADS) factor_kernel(Dims dm, Ws ws) {
  extern __shared__ float fsm[];
  float* A = fsm;               // [D][FA_LD]: A, then L in the lower triangle
  float* X = fsm + D * FA_LD;   // [D][FA_LD]: L^{-1}
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

  // G = sum of partials in chunk order; A = I + G
  const float* gp = ws.gpart + ((int64_t)plane * dm.c_cap) * D * D;
  float* gout = ws.gram + (int64_t)u * D * D;
  for (int e = tid; e < D * D; e += FA_THREADS) {
    float acc = 0.f;
    for (int c = c0; c < c1; ++c) acc += gp[(int64_t)c * D * D + e];
    gout[e] = acc;
    const int r = e / D, c = e % D;
    A[r * FA_LD + c] = acc + (r == c ? 1.f : 0.f);
  }
  __syncthreads();

  // Cholesky A = L L^T (lower triangle of A overwritten by L)
  for (int j = 0; j < D; ++j) {
    if (tid == 0) {
      const float djj = A[j * FA_LD + j];
      if (!(djj > 0.f) || !isfinite(djj)) s_bad = 1;
      A[j * FA_LD + j] = sqrtf(fmaxf(djj, 1e-30f));
    }
    __syncthreads();
    const float ljj = A[j * FA_LD + j];
    for (int i = j + 1 + tid; i < D; i += FA_THREADS) A[i * FA_LD + j] /= ljj;
    __syncthreads();
    const int n = D - 1 - j;
    for (int e = tid; e < n * n; e += FA_THREADS) {
      const int ii = j + 1 + e / n, kk = j + 1 + e % n;
      if (kk <= ii) A[ii * FA_LD + kk] -= A[ii * FA_LD + j] * A[kk * FA_LD + j];
    }
    __syncthreads();
  }

  // L^{-1}: thread j solves L x = e_j (column j), x_i = 0 for i < j
  if (tid < D) {
    const int j = tid;
    for (int i = 0; i < j; ++i) X[i * FA_LD + j] = 0.f;
    X[j * FA_LD + j] = 1.f / A[j * FA_LD + j];
    for (int i = j + 1; i < D; ++i) {
      float acc = 0.f;
      for (int k = j; k < i; ++k) acc = fmaf(A[i * FA_LD + k], X[k * FA_LD + j], acc);
      X[i * FA_LD + j] = -acc / A[i * FA_LD + i];
    }
  }
  __syncthreads();

  float* mout = ws.minv + (int64_t)u * D * D;
  for (int e = tid; e < D * D; e += FA_THREADS) {
    const int r = e / D, c = e % D;
    const float x = X[r * FA_LD + c];
    mout[e] = x;
    if (!isfinite(x)) s_bad = 1;
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
      const float x0 = X[r * FA_LD + cc * 8 + 2 * q];
      const float x1 = X[r * FA_LD + cc * 8 + 2 * q + 1];
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
