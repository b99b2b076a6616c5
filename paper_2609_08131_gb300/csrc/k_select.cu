// k_select.cu - TOP-B selection (Algorithm 1 step 5) and compaction of the
// retained cache Z_C (Sec. 3.1).
//
// select_kernel: one 1024-thread CTA per unit (grid-stride). Scores are
// non-negative float32, so their bit patterns order like unsigned integers.
// Four 8-bit radix passes (most significant digit first, shared-memory
// histograms) find the B-th largest key T and how many keys equal to T are
// still needed; one ordered pass then keeps every key > T and the first
// `need` keys == T by position (ties go to the lower position), writing the
// kept positions in ascending order through block-wide ballot scans. All of
// it is deterministic.
//
// compact_kernel: 16-byte vector copies of the kept K and V rows into the
// dense [L][Hkv][S][B][d] output; rows of -1 (or of a position outside the
// request) are zero-filled, so no index value can make it read out of bounds.
#include "jacap_dev.cuh"
#include "jacap_internal.h"

namespace jacap {

constexpr int SE_THREADS = 1024;

// Exclusive block-wide prefix count of `pred`; returns the prefix for this
// thread and writes the block total to *total. Uses wsum[32] in smem.
__device__ __forceinline__ int block_excl_count(bool pred, int* wsum, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned bal = __ballot_sync(0xffffffffu, pred);
  const int in_warp = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) wsum[warp] = __popc(bal);
  __syncthreads();
  if (warp == 0) {
    const int x = wsum[lane];
    int incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    wsum[lane] = incl - x;  // exclusive
    if (lane == 31) wsum[32] = incl;
  }
  __syncthreads();
  const int r = wsum[warp] + in_warp;
  *total = wsum[32];
  __syncthreads();
  return r;
}

__global__ void __launch_bounds__(SE_THREADS)
    select_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu, const float* __restrict__ scores, int B,
                  int32_t* __restrict__ idx, int32_t* __restrict__ kept) {
  __shared__ uint32_t hist[256];
  __shared__ int wsum[33];
  __shared__ uint32_t s_digit, s_need;
  __shared__ int s_skip;
  const int tid = threadIdx.x;
  if (tid == 0) s_skip = status_failed(ws) ? 1 : 0;
  __syncthreads();
  if (s_skip) return;
  const int units = dm.L * dm.Hkv * dm.S;
  for (int u = blockIdx.x; u < units; u += gridDim.x) {
    const int plane = u / dm.S, s = u % dm.S;
    const int64_t start = cu[s];
    const int64_t end = cu[s + 1];
    int32_t* out = idx + (int64_t)u * B;
    if (start < 0 || end < start || end > dm.Ntot) {  // malformed cu_seqlens: no reads
      for (int r = tid; r < B; r += SE_THREADS) out[r] = -1;
      if (tid == 0) {
        flag(ws, ST_INVALID);
        if (plane == 0) kept[s] = 0;
      }
      continue;
    }
    const int n = (int)(end - start);
    const uint32_t* key = (const uint32_t*)(scores + (int64_t)plane * dm.Ntot + start);
    if (plane == 0 && tid == 0) kept[s] = min(n, B);
    if (n <= B) {
      for (int r = tid; r < B; r += SE_THREADS) out[r] = r < n ? r : -1;
      continue;
    }
    // ---- radix select of the B-th largest key ----
    uint32_t prefix = 0, mask = 0, need = (uint32_t)B;
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int b = tid; b < 256; b += SE_THREADS) hist[b] = 0;
      __syncthreads();
      for (int i = tid; i < n; i += SE_THREADS) {
        const uint32_t k = key[i];
        if ((k & mask) == prefix) atomicAdd(&hist[(k >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (tid == 0) {
        uint32_t above = 0;
        int d = 255;
        for (; d > 0; --d) {
          if (above + hist[d] >= need) break;
          above += hist[d];
        }
        s_digit = (uint32_t)d;
        s_need = need - above;
      }
      __syncthreads();
      prefix |= s_digit << shift;
      mask |= 255u << shift;
      need = s_need;
      __syncthreads();
    }
    const uint32_t T = prefix;  // the B-th largest key; `need` keys == T are kept
    // ---- ordered emission ----
    int written = 0, eq_seen = 0;
    for (int base = 0; base < n && written < B; base += SE_THREADS) {
      const int i = base + tid;
      const uint32_t k = i < n ? key[i] : 0u;
      const bool gt = i < n && k > T;
      const bool eq = i < n && k == T;
      int eq_total;
      const int eq_rank = eq_seen + block_excl_count(eq, wsum, &eq_total);
      const bool sel = gt || (eq && eq_rank < (int)need);
      int sel_total;
      const int pos = written + block_excl_count(sel, wsum, &sel_total);
      if (sel && pos < B) out[pos] = i;
      written += sel_total;
      eq_seen += eq_total;
    }
    __syncthreads();
  }
}

template <typename T>
__global__ void __launch_bounds__(256)
    compact_kernel(Dims dm, const int32_t* __restrict__ cu, const T* __restrict__ k, const T* __restrict__ v,
                   const int32_t* __restrict__ idx, int B, T* __restrict__ k_out, T* __restrict__ v_out) {
  constexpr int CH = D * (int)sizeof(T) / 16;  // 16-byte chunks per row
  const int64_t rows = (int64_t)dm.L * dm.Hkv * dm.S * B;
  const int64_t total = rows * CH;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = e / CH;
    const int c = (int)(e % CH);
    const int64_t u = row / B;
    const int plane = (int)(u / dm.S), s = (int)(u % dm.S);
    const int l = plane / dm.Hkv, g = plane % dm.Hkv;
    const int32_t src = idx[row];
    const int64_t start = cu[s], end = cu[s + 1];
    uint4 kk = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
    // positions outside the request (or a malformed cu_seqlens) give zero rows
    if (src >= 0 && start >= 0 && start + src < end && end <= dm.Ntot) {
      const int64_t off = (int64_t)l * dm.kv_sl + (int64_t)g * dm.kv_sh + ((int64_t)cu[s] + src) * dm.kv_st;
      kk = *((const uint4*)(k + off) + c);
      vv = *((const uint4*)(v + off) + c);
    }
    *((uint4*)(k_out + row * D) + c) = kk;
    *((uint4*)(v_out + row * D) + c) = vv;
  }
}

cudaError_t launch_select(const Dims& dm, const Ws& ws, const int32_t* cu, const float* scores, int budget,
                          int32_t* idx, int32_t* kept, int grid, cudaStream_t st) {
  select_kernel<<<grid, SE_THREADS, 0, st>>>(dm, ws, cu, scores, budget, idx, kept);
  return cudaGetLastError();
}

cudaError_t launch_compact(const Dims& dm, int dtype, const int32_t* cu, const void* k, const void* v,
                           const int32_t* idx, int budget, void* k_out, void* v_out, cudaStream_t st) {
  const int64_t rows = (int64_t)dm.L * dm.Hkv * dm.S * budget;
  const int es = dtype == 1 ? 2 : 4;
  const int64_t total = rows * (D * es / 16);
  const int64_t blocks64 = (total + 255) / 256;
  const int blocks = (int)(blocks64 < 65535 * 16 ? blocks64 : 65535 * 16);
  if (blocks <= 0) return cudaSuccess;
  if (dtype == 1)
    compact_kernel<__nv_bfloat16><<<blocks, 256, 0, st>>>(dm, cu, (const __nv_bfloat16*)k, (const __nv_bfloat16*)v,
                                                          idx, budget, (__nv_bfloat16*)k_out, (__nv_bfloat16*)v_out);
  else
    compact_kernel<float><<<blocks, 256, 0, st>>>(dm, cu, (const float*)k, (const float*)v, idx, budget,
                                                  (float*)k_out, (float*)v_out);
  return cudaGetLastError();
}

}  // namespace jacap
