// k_decode.cu - the pieces of decoding-stage eviction that the prefill pass
// does not already have.
//
// During decoding the query statistics are estimated from the queries seen so
// far (Sec. 3.4, last paragraph), not from a fixed window: every decode step
// adds one query per (request, layer, query head). The running statistics are
// kept as (count n, mean m, sum of squared deviations M2) per channel and a
// batch of new queries is merged with the pairwise update of Chan, Golub and
// LeVeque (1979):
//   n = n_a + n_b,  delta = m_b - m_a,  m = m_a + delta n_b / n,
//   M2 = M2_a + M2_b + delta^2 n_a n_b / n,
// with (m_b, M2_b) of the batch taken in two passes. At an eviction the
// scoring pass reads mu = m and lambda = M2 / n (or M2 / (n - 1)) instead of
// window statistics.
//
// After the TOP-B selection the cache of a request is compacted in place so
// that the kept rows occupy rows 0 .. kept - 1 of the request's range, in one
// of two ways (one CTA per unit in both; jacap_inplace.cuh holds the per-unit
// code, which the selection kernel also runs right after selecting a unit):
//  - ascending order (the order of jacap_compact): every kept row moves to
//    its rank. The rows move in chunks; every chunk is read completely before
//    any of it is written (a barrier in between). Because the kept positions
//    ascend strictly from 0, idx[r] >= r, so a chunk's writes (rows c0 ..
//    c0 + CH - 1) never touch a row that a later chunk still has to read
//    (rows >= c0 + CH). Up to `kept` rows move.
//  - hole filling: kept rows below `kept` stay where they are; the kept rows
//    at or above `kept` move, in ascending order, into the evicted rows below
//    `kept`, in ascending order. Sources and destinations are disjoint, so all
//    copies run at once, and at most n - kept rows move (the eviction interval
//    during decoding, instead of the whole budget). If f kept positions lie
//    below `kept`, the evicted row r between the (i-1)-th and i-th of them is
//    hole number r - i and receives row idx[f + r - i].
#include "jacap_dev.cuh"
#include "jacap_inplace.cuh"
#include "jacap_internal.h"

namespace jacap {

template <typename T>
__device__ __forceinline__ float q_elem(const T* p);
template <>
__device__ __forceinline__ float q_elem<float>(const float* p) { return __ldg(p); }
template <>
__device__ __forceinline__ float q_elem<__nv_bfloat16>(const __nv_bfloat16* p) { return __bfloat162float(*p); }

// One block per (request, layer, query head); thread c owns channel c.
// stats: [S][L][Hq][2][D] (mean, M2); counts: [S][L][Hq].
template <typename T>
__global__ void __launch_bounds__(D)
    stats_update_kernel(Dims dm, const T* __restrict__ q, float* stats, int32_t* counts, int reset) {
  pdl_wait();
  const int b = blockIdx.x;
  const int h = b % dm.Hq;
  const int l = (b / dm.Hq) % dm.L;
  const int s = b / (dm.Hq * dm.L);
  const int c = threadIdx.x;
  const T* base = q + (int64_t)s * dm.q_ss + (int64_t)l * dm.q_sl + (int64_t)h * dm.q_sh + c;
  const int nb = dm.window;
  float sum = 0.f;
  for (int j = 0; j < nb; ++j) sum += q_elem(base + (int64_t)j * dm.q_sp);
  const float mb = sum / (float)nb;
  float m2b = 0.f;
  for (int j = 0; j < nb; ++j) {
    const float e = q_elem(base + (int64_t)j * dm.q_sp) - mb;
    m2b = fmaf(e, e, m2b);
  }
  float* st = stats + (int64_t)b * 2 * D;
  int na = reset ? 0 : counts[b];
  if (na < 0) na = 0;
  float mean = mb, m2 = m2b;
  if (na > 0) {
    const float n = (float)na + (float)nb;
    const float ma = st[c], delta = mb - ma;
    mean = fmaf(delta, (float)nb / n, ma);
    m2 = st[D + c] + m2b + delta * delta * ((float)na * (float)nb / n);
  }
  __syncthreads();  // every thread has read counts[b] before it changes
  st[c] = mean;
  st[D + c] = m2;
  if (c == 0) counts[b] = na + nb;
}

// The scoring pass's query statistics from running statistics: the same
// outputs as the window statistics (mu / (tau sqrt d) and lambda).
__global__ void __launch_bounds__(D)
    stats_moments_kernel(Dims dm, Ws ws, const float* __restrict__ stats, const int32_t* __restrict__ counts) {
  pdl_wait();
  if (status_failed(ws)) return;
  const int b = blockIdx.x, c = threadIdx.x;
  const int n = counts[b];
  if (n < (dm.cov_unbiased ? 2 : 1)) {
    if (c == 0) flag(ws, ST_INVALID);
    return;
  }
  const float mean = stats[(int64_t)b * 2 * D + c];
  const float lam = stats[(int64_t)b * 2 * D + D + c] / (float)(dm.cov_unbiased ? n - 1 : n);
  ws.mu[(int64_t)b * D + c] = mean * dm.inv_scale;
  ws.lam[(int64_t)b * D + c] = lam;
  if (!isfinite(mean) || !isfinite(lam) || lam < 0.f) flag(ws, ST_NONFINITE);
}

constexpr int CI_THREADS = 256;

// One CTA per unit u = (l Hkv + g) S + s, the order of jacap_select's idx. The
// kept positions come from the caller: a unit whose positions do not ascend
// strictly within [0, n) is left untouched and flagged.
template <typename T>
__global__ void __launch_bounds__(CI_THREADS)
    compact_inplace_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu, T* k, T* v, int32_t* pos,
                           const int32_t* __restrict__ idx, int budget) {
  pdl_wait();
  if (status_failed(ws)) return;
  const int u = blockIdx.x;
  const int s = u % dm.S, plane = u / dm.S;
  const int tid = threadIdx.x;
  const int64_t t0 = cu[s];
  const int64_t n = (int64_t)cu[s + 1] - t0;
  const int kept = (int)(n < (int64_t)budget ? n : (int64_t)budget);
  const int32_t* ix = idx + (int64_t)u * budget;
  int bad = 0;
  for (int r = tid; r < kept; r += CI_THREADS) {
    const int32_t x = ix[r];
    bad |= x < 0 || (int64_t)x >= n || (r > 0 && x <= ix[r - 1]);
  }
  if (__syncthreads_or(bad)) {
    if (tid == 0) flag(ws, ST_INVALID);
    return;
  }
  compact_ordered_unit<T, CI_THREADS>(dm, plane, t0, kept, k, v, pos, ix);
}

template <typename T>
__global__ void __launch_bounds__(CI_THREADS)
    fill_holes_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu, T* k, T* v, int32_t* pos,
                      const int32_t* __restrict__ idx, int budget) {
  pdl_wait();
  __shared__ int s_f;
  if (status_failed(ws)) return;
  const int u = blockIdx.x;
  const int s = u % dm.S, plane = u / dm.S;
  const int tid = threadIdx.x;
  const int64_t t0 = cu[s];
  const int64_t n = (int64_t)cu[s + 1] - t0;
  const int kept = (int)(n < (int64_t)budget ? n : (int64_t)budget);
  const int32_t* ix = idx + (int64_t)u * budget;
  if (tid == 0) s_f = 0;
  __syncthreads();
  int bad = 0;
  for (int r = tid; r < kept; r += CI_THREADS) {
    const int32_t x = ix[r];
    bad |= x < 0 || (int64_t)x >= n || (r > 0 && x <= ix[r - 1]);
    // f = the number of kept positions below `kept`
    if (x < kept && (r + 1 == kept || ix[r + 1] >= kept)) s_f = r + 1;
  }
  if (__syncthreads_or(bad)) {
    if (tid == 0) flag(ws, ST_INVALID);
    return;
  }
  fill_holes_unit<T, CI_THREADS>(dm, plane, t0, kept, s_f, k, v, pos, ix);
}

template <typename T>
static cudaError_t launch_stats_update_t(const Dims& dm, const void* q, float* stats, int32_t* counts, int reset,
                                         cudaStream_t st) {
  JACAP_TRY(launch_pdl(dm.pdl != 0, stats_update_kernel<T>, dm.S * dm.L * dm.Hq, D, 0, st, dm, (const T*)q, stats,
                       counts, reset));
  return cudaGetLastError();
}

cudaError_t launch_stats_update(const Dims& dm, int dtype, const void* q, float* stats, int32_t* counts, int reset,
                                cudaStream_t st) {
  return dtype == 1 ? launch_stats_update_t<__nv_bfloat16>(dm, q, stats, counts, reset, st)
                    : launch_stats_update_t<float>(dm, q, stats, counts, reset, st);
}

cudaError_t launch_stats_moments(const Dims& dm, const Ws& ws, const float* stats, const int32_t* counts,
                                 cudaStream_t st) {
  JACAP_TRY(launch_pdl(dm.pdl != 0, stats_moments_kernel, dm.S * dm.L * dm.Hq, D, 0, st, dm, ws, stats, counts));
  return cudaGetLastError();
}

cudaError_t launch_compact_inplace(const Dims& dm, const Ws& ws, int dtype, const int32_t* cu, void* k, void* v,
                                   int32_t* pos, const int32_t* idx, int budget, int preserve_order,
                                   cudaStream_t st) {
  const int units = dm.L * dm.Hkv * dm.S;
  if (!preserve_order) {
    if (dtype == 1)
      JACAP_TRY(launch_pdl(dm.pdl != 0, fill_holes_kernel<__nv_bfloat16>, units, CI_THREADS, 0, st, dm, ws, cu,
                           (__nv_bfloat16*)k, (__nv_bfloat16*)v, pos, idx, budget));
    else
      JACAP_TRY(launch_pdl(dm.pdl != 0, fill_holes_kernel<float>, units, CI_THREADS, 0, st, dm, ws, cu, (float*)k,
                           (float*)v, pos, idx, budget));
    return cudaGetLastError();
  }
  if (dtype == 1)
    JACAP_TRY(launch_pdl(dm.pdl != 0, compact_inplace_kernel<__nv_bfloat16>, units, CI_THREADS, 0, st, dm, ws, cu,
                         (__nv_bfloat16*)k, (__nv_bfloat16*)v, pos, idx, budget));
  else
    JACAP_TRY(launch_pdl(dm.pdl != 0, compact_inplace_kernel<float>, units, CI_THREADS, 0, st, dm, ws, cu, (float*)k,
                         (float*)v, pos, idx, budget));
  return cudaGetLastError();
}

}  // namespace jacap
