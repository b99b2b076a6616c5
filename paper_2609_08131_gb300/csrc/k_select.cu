// k_select.cu - TOP-B selection (Algorithm 1 step 5) and compaction of the
// retained cache Z_C (Sec. 3.1).
//
// select_kernel: one CTA per unit (grid-stride), of NT = 1024 threads, or of
// 256 when the longest request has at most 4096 tokens and there are more
// units than SMs (then four or more CTAs fit an SM and a pass over many short
// units, as in decoding-stage eviction, runs in one wave), or of 512 (two per
// SM) for longer requests when there are more than two SMs' worth of units. Scores are
// non-negative float32, so their bit patterns order like unsigned integers.
// Three radix passes (digits of 11, 11 and 10 bits, most significant first,
// shared-memory histograms; a pass counts only keys that match the digits
// found so far) find the B-th largest key T and how many keys equal to T are
// still needed. The keys are read in slabs of NT KPT into registers (KPT
// per lane, all loads in flight together; KPT = 4, 8, 16 or 32, the smallest
// that holds the longest request in one slab); a request that fits one slab is
// read once and every pass works on registers. Emission walks the slabs in
// order; in a slab each warp owns 32 KPT consecutive positions, counts its keys
// > T and == T with ballots, and the warp totals give where its kept
// positions go and which of its keys == T are among the first `need` by
// position (ties go to the lower position); kept positions come out in
// ascending order. All of it is deterministic.
//
// compact_kernel: 16-byte vector copies of the kept K and V rows into the
// dense [L][Hkv][S][B][d] output; rows of -1 (or of a position outside the
// request) are zero-filled, so no index value can make it read out of bounds.
//
// select_kernel can also finish each unit itself as soon as its positions are
// emitted, so the rows move while other CTAs are still selecting and no
// separate compaction launch follows: MODE 1 copies the kept rows into k_out,
// v_out (the work of compact_kernel, same zero fill); MODE 2 fills the holes
// of the cache in place (jacap_inplace.cuh, as jacap_compact_inplace does).
// MODE 0 only selects. (The in-place compaction in ascending order moves
// every kept row; it stays a launch of its own, whose small CTAs keep more
// bytes in flight per SM than one selection CTA per unit could.)
#include "jacap_dev.cuh"
#include "jacap_inplace.cuh"
#include "jacap_internal.h"

namespace jacap {


constexpr int SE_BINS = 2048;

// Keys of slab `sl` into registers: lane's register j holds position
// sl * NT KPT + 32 KPT w + 32 j + lane (coalesced; all loads in flight at
// once). KPT keys per lane (4 .. 32) is chosen from the longest request, so a
// short cache does not carry empty register slots through every pass.
template <int KPT, int NT>
__device__ __forceinline__ void load_slab(const uint32_t* key, int n, int sl, int warp, int lane,
                                          uint32_t (&kr)[KPT]) {
  const int base = sl * NT * KPT + warp * (32 * KPT) + lane;
#pragma unroll
  for (int j = 0; j < KPT; ++j) {
    const int i = base + 32 * j;
    kr[j] = i < n ? __ldg(key + i) : 0u;
  }
}

// Rows out[0 .. B) of unit u (positions relative to the request start, as
// emitted) from K and V into k_out, v_out; -1 or a position outside the
// request gives a zero row. All threads of the CTA; out was written by them
// before the barrier that precedes this call.
template <typename T, int NT>
__device__ __forceinline__ void gather_unit(const Dims& dm, int plane, int64_t start, int64_t end, bool valid,
                                            const T* __restrict__ k, const T* __restrict__ v,
                                            const int32_t* out, int B, int64_t u, T* __restrict__ k_out,
                                            T* __restrict__ v_out) {
  constexpr int CH = D * (int)sizeof(T) / 16;  // 16-byte chunks per row
  const int l = plane / dm.Hkv, g = plane % dm.Hkv;
  const int64_t base = (int64_t)l * dm.kv_sl + (int64_t)g * dm.kv_sh;
  uint4* ko = (uint4*)(k_out + u * B * D);
  uint4* vo = (uint4*)(v_out + u * B * D);
#pragma unroll 4
  for (int e = threadIdx.x; e < B * CH; e += NT) {
    const int r = e / CH, c = e % CH;
    const int32_t src = out[r];
    uint4 kk = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
    if (valid && src >= 0 && start + src < end) {
      const int64_t off = base + (start + src) * dm.kv_st;
      kk = *((const uint4*)(k + off) + c);
      vv = *((const uint4*)(v + off) + c);
    }
    ko[e] = kk;
    vo[e] = vv;
  }
}

template <int KPT, typename E, int MODE, int NT>
__global__ void __launch_bounds__(NT, NT == 512 ? 2 : 1)
    select_kernel(Dims dm, Ws ws, const int32_t* __restrict__ cu, const float* __restrict__ scores, int B,
                  int32_t* __restrict__ idx, int32_t* __restrict__ kept, const E* __restrict__ k,
                  const E* __restrict__ v, E* __restrict__ k_out, E* __restrict__ v_out, E* kio, E* vio,
                  int32_t* pos) {
  constexpr bool GATHER = MODE == 1;
  pdl_wait();
  constexpr int SE_KPT = KPT;
  constexpr int SE_SLAB = NT * KPT;  // warp w holds positions 32 KPT w .. + 32 KPT - 1 of a slab
  constexpr int NW = NT / 32;
  __shared__ uint32_t hist[SE_BINS];
  __shared__ uint32_t s_digit, s_need;
  __shared__ int s_skip;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) s_skip = status_failed(ws) ? 1 : 0;
  __syncthreads();
  if (s_skip) return;
  const int units = dm.L * dm.Hkv * dm.S;
  const uint32_t lt = (1u << lane) - 1u;
  // time accounting (trace builds, thread 0): 0 the scores loaded (one slab),
  // 1 the radix passes, 2 the emission, 3 the rows gathered, 4 units, 5 the
  // whole unit (units of more than B tokens)
  TRC_DECL(TR_CTA_SLOTS);
  for (int u = blockIdx.x; u < units; u += gridDim.x) {
    TRC_T(tr_u);
    const int plane = u / dm.S, s = u % dm.S;
    const int64_t start = cu[s];
    const int64_t end = cu[s + 1];
    int32_t* out = idx + (int64_t)u * B;
    const bool valid = !(start < 0 || end < start || end > dm.Ntot);
    if (!valid) {  // malformed cu_seqlens: no reads
      for (int r = tid; r < B; r += NT) out[r] = -1;
      if (tid == 0) {
        flag(ws, ST_INVALID);
        if (plane == 0) kept[s] = 0;
      }
      if constexpr (GATHER) {
        __syncthreads();
        gather_unit<E, NT>(dm, plane, start, end, false, k, v, out, B, u, k_out, v_out);
      }
      continue;
    }
    const int n = (int)(end - start);
    const uint32_t* key = (const uint32_t*)(scores + (int64_t)plane * dm.Ntot + start);
    if (plane == 0 && tid == 0) kept[s] = min(n, B);
    if (n <= B) {
      for (int r = tid; r < B; r += NT) out[r] = r < n ? r : -1;
      if constexpr (GATHER) {
        __syncthreads();
        gather_unit<E, NT>(dm, plane, start, end, true, k, v, out, B, u, k_out, v_out);
      }
      continue;
    }
    const int nslab = (n + SE_SLAB - 1) / SE_SLAB;
    uint32_t kr[SE_KPT];
    TRC_INC(4);
    if (nslab == 1) load_slab<KPT, NT>(key, n, 0, warp, lane, kr);  // register-resident for all passes
    TRC_ADD(0, tr_u);
    TRC_T(tr_r);
    // ---- radix select of the B-th largest key: digits [31:21], [20:10], [9:0] ----
    uint32_t prefix = 0, mask = 0, need = (uint32_t)B;
#pragma unroll 1
    for (int pass = 0; pass < 3; ++pass) {
      const int shift = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
      const uint32_t dmask = pass == 2 ? 1023u : 2047u;
      for (int b = tid; b < SE_BINS; b += NT) hist[b] = 0;
      __syncthreads();
#pragma unroll 1
      for (int sl = 0; sl < nslab; ++sl) {
        if (nslab > 1) load_slab<KPT, NT>(key, n, sl, warp, lane, kr);
        const int base = sl * SE_SLAB + warp * (32 * SE_KPT) + lane;
#pragma unroll
        for (int j = 0; j < SE_KPT; ++j)
          if (base + 32 * j < n && (kr[j] & mask) == prefix) atomicAdd(&hist[(kr[j] >> shift) & dmask], 1u);
      }
      __syncthreads();
      if (warp == 0) {
        // lane l sums bins 64 l .. 64 l + 63 (in a rotated order, so that the
        // lanes' loads fall in different banks); suffix sums over the lanes
        // locate the group of 64 bins that holds the need-th largest key, and
        // a second suffix scan over that group (two bins per lane) the bin
        uint32_t c = 0;
#pragma unroll 8
        for (int b = 0; b < 64; ++b) c += hist[64 * lane + ((b + lane) & 63)];
        uint32_t suf = c;  // sum over lanes >= lane
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_down_sync(0xffffffffu, suf, o);
          if (lane + o < 32) suf += y;
        }
        const uint32_t above = suf - c;  // keys in bins of higher lanes
        const uint32_t hit = __ballot_sync(0xffffffffu, above < need && suf >= need);  // exactly one lane
        const int g = __ffs(hit) - 1;
        const uint32_t gabove = __shfl_sync(0xffffffffu, above, g);  // keys above the group
        // bins 64 g + 2 lane (+1), suffix sums from the top of the group down
        const uint32_t h0 = hist[64 * g + 2 * lane], h1 = hist[64 * g + 2 * lane + 1];
        const uint32_t c2 = h0 + h1;
        uint32_t suf2 = c2;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_down_sync(0xffffffffu, suf2, o);
          if (lane + o < 32) suf2 += y;
        }
        const uint32_t a1 = gabove + suf2 - c2;  // keys above bin 2 lane + 1 of the group
        const uint32_t a0 = a1 + h1;             // keys above bin 2 lane
        // the bin d with (keys above d) < need <= (keys above d) + hist[d]
        const bool in1 = a1 < need && a1 + h1 >= need, in0 = a0 < need && a0 + h0 >= need;
        if (in1) {
          s_digit = (uint32_t)(64 * g + 2 * lane + 1);
          s_need = need - a1;
        } else if (in0) {
          s_digit = (uint32_t)(64 * g + 2 * lane);
          s_need = need - a0;
        }
      }
      __syncthreads();
      prefix |= s_digit << shift;
      mask |= dmask << shift;
      need = s_need;
      __syncthreads();
    }
    const uint32_t T = prefix;  // the B-th largest key; the first `need` keys == T are kept
    TRC_ADD(1, tr_r);
    TRC_T(tr_e);
    // ---- emission, slab by slab; in a slab warp w owns positions 32 KPT w .. ----
    uint32_t gt_run = 0, eq_run = 0;  // kept-greater and equal keys before this slab
#pragma unroll 1
    for (int sl = 0; sl < nslab; ++sl) {
      if (nslab > 1) load_slab<KPT, NT>(key, n, sl, warp, lane, kr);
      const int base = sl * SE_SLAB + warp * (32 * SE_KPT) + lane;
      // the warp's counts of keys > T and == T, and which register slots hold
      // any key >= T (most hold none: only B of the n keys are kept)
      uint32_t gt = 0, eq = 0, jmask = 0;
#pragma unroll
      for (int j = 0; j < SE_KPT; ++j) {
        const bool v = base + 32 * j < n;
        const uint32_t bg = __ballot_sync(0xffffffffu, v && kr[j] > T);
        const uint32_t be = __ballot_sync(0xffffffffu, v && kr[j] == T);
        gt += __popc(bg);
        eq += __popc(be);
        if (bg | be) jmask |= 1u << j;
      }
      if (lane == 0) {
        hist[warp] = gt;  // the histogram is free again: it holds the warp totals
        hist[NW + warp] = eq;
      }
      __syncthreads();
      if (warp == 0) {  // exclusive prefixes of the warp totals (lane w: warp w) and the slab totals
        const uint32_t g = lane < NW ? hist[lane] : 0u, e = lane < NW ? hist[NW + lane] : 0u;
        uint32_t gs = g, es = e;  // inclusive scans
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_up_sync(0xffffffffu, gs, o), z = __shfl_up_sync(0xffffffffu, es, o);
          if (lane >= o) {
            gs += y;
            es += z;
          }
        }
        if (lane < NW) {
          hist[2 * NW + lane] = gs - g;
          hist[3 * NW + lane] = es - e;
        }
        if (lane == 31) {
          hist[4 * NW] = gs;
          hist[4 * NW + 1] = es;
        }
      }
      __syncthreads();
      const uint32_t gt_before = gt_run + hist[2 * NW + warp], eq_before = eq_run + hist[3 * NW + warp];
      const uint32_t gt_all = hist[4 * NW], eq_all = hist[4 * NW + 1];
      // kept before this warp's block: all greater keys plus the equal ones of rank < need
      uint32_t pos = gt_before + min(eq_before, need);
      uint32_t er = eq_before;
#pragma unroll
      for (int j = 0; j < SE_KPT; ++j) {
        if (!(jmask & (1u << j))) continue;  // warp-uniform: no key >= T in this slot
        const int i = base + 32 * j;
        const bool v = i < n;
        const uint32_t beq = __ballot_sync(0xffffffffu, v && kr[j] == T);
        const uint32_t my_er = er + __popc(beq & lt);
        const bool sel = v && (kr[j] > T || (kr[j] == T && my_er < need));
        const uint32_t bsel = __ballot_sync(0xffffffffu, sel);
        const uint32_t my_pos = pos + __popc(bsel & lt);
        if (sel && my_pos < (uint32_t)B) out[my_pos] = i;
        pos += __popc(bsel);
        er += __popc(beq);
      }
      gt_run += gt_all;
      eq_run += eq_all;
      __syncthreads();  // the totals in hist are read before the next slab rewrites them
    }
    // (the barrier that ends the last slab also orders the emitted positions
    // before they are read back here)
    TRC_ADD(2, tr_e);
    TRC_T(tr_g);
    if constexpr (GATHER) gather_unit<E, NT>(dm, plane, start, end, true, k, v, out, B, u, k_out, v_out);
    TRC_ADD(3, tr_g);
    if constexpr (MODE == 2) {
      // f = the kept positions below B (they ascend: a binary search)
      int lo = 0, hi = B;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (out[mid] < B) lo = mid + 1; else hi = mid;
      }
      fill_holes_unit<E, NT>(dm, plane, start, B, lo, kio, vio, pos, out);
    }
    if constexpr (MODE == 2) __syncthreads();  // the unit's rows have moved before `out` is reused
    TRC_ADD(5, tr_u);
  }
  if (tid == 0) TRC_PUT(ws, TR_K_SELECT, 6);
}

template <typename T>
__global__ void __launch_bounds__(256)
    compact_kernel(Dims dm, const int32_t* __restrict__ cu, const T* __restrict__ k, const T* __restrict__ v,
                   const int32_t* __restrict__ idx, int B, T* __restrict__ k_out, T* __restrict__ v_out) {
  pdl_wait();
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

template <int KPT, int NT>
static cudaError_t launch_select_kpt(const Dims& dm, const Ws& ws, const int32_t* cu, const float* scores, int budget,
                                     int32_t* idx, int32_t* kept, int dtype, const void* k, const void* v,
                                     void* k_out, void* v_out, void* kio, void* vio, int32_t* pos, int grid,
                                     cudaStream_t st) {
  using bf = __nv_bfloat16;
  if (kio != nullptr) {  // hole filling in place
    if (dtype == 1)
      return launch_pdl(dm.pdl != 0, select_kernel<KPT, bf, 2, NT>, grid, NT, 0, st, dm, ws, cu, scores, budget,
                        idx, kept, (const bf*)nullptr, (const bf*)nullptr, (bf*)nullptr, (bf*)nullptr, (bf*)kio,
                        (bf*)vio, pos);
    return launch_pdl(dm.pdl != 0, select_kernel<KPT, float, 2, NT>, grid, NT, 0, st, dm, ws, cu, scores, budget,
                      idx, kept, (const float*)nullptr, (const float*)nullptr, (float*)nullptr, (float*)nullptr,
                      (float*)kio, (float*)vio, pos);
  }
  if (k == nullptr)
    return launch_pdl(dm.pdl != 0, select_kernel<KPT, bf, 0, NT>, grid, NT, 0, st, dm, ws, cu, scores, budget,
                      idx, kept, (const bf*)nullptr, (const bf*)nullptr, (bf*)nullptr, (bf*)nullptr, (bf*)nullptr,
                      (bf*)nullptr, (int32_t*)nullptr);
  if (dtype == 1)
    return launch_pdl(dm.pdl != 0, select_kernel<KPT, bf, 1, NT>, grid, NT, 0, st, dm, ws, cu, scores, budget,
                      idx, kept, (const bf*)k, (const bf*)v, (bf*)k_out, (bf*)v_out, (bf*)nullptr, (bf*)nullptr,
                      (int32_t*)nullptr);
  return launch_pdl(dm.pdl != 0, select_kernel<KPT, float, 1, NT>, grid, NT, 0, st, dm, ws, cu, scores, budget,
                    idx, kept, (const float*)k, (const float*)v, (float*)k_out, (float*)v_out, (float*)nullptr,
                    (float*)nullptr, (int32_t*)nullptr);
}

cudaError_t launch_select(const Dims& dm, const Ws& ws, const int32_t* cu, const float* scores, int budget,
                          int32_t* idx, int32_t* kept, int max_seqlen, int grid, cudaStream_t st, int dtype,
                          const void* k, const void* v, void* k_out, void* v_out, void* kio, void* vio,
                          int32_t* pos) {
#define JACAP_SELECT(KPT, NT)                                                                                   \
  JACAP_TRY((launch_select_kpt<KPT, NT>(dm, ws, cu, scores, budget, idx, kept, dtype, k, v, k_out, v_out, kio, vio, \
                                        pos, grid, st)))
  // small CTAs only pay off when the 1024-thread ones would need more than one
  // wave (one per SM fits); for a few units the larger CTA finishes each sooner
  int dev = 0, sms = 0;
  JACAP_TRY(cudaGetDevice(&dev));
  JACAP_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const int64_t units = (int64_t)dm.L * dm.Hkv * dm.S;
  const bool small = units > sms;
  if (small && max_seqlen <= 256 * 4) JACAP_SELECT(4, 256);
  else if (small && max_seqlen <= 256 * 8) JACAP_SELECT(8, 256);
  else if (small && max_seqlen <= 256 * 16) JACAP_SELECT(16, 256);
  // more than two waves of 1024-thread CTAs: two 512-thread CTAs per SM (keys
  // in slabs of 16384, re-read from L2 by each pass) keep twice as many units
  // going (config 5's 4096 units: 0.95 -> 0.85 ms); with fewer units the
  // larger CTA finishes each unit sooner (256 units of 131072 tokens: 0.159
  // against 0.170 ms)
  else if (units > 2 * (int64_t)sms && max_seqlen > 1024 * 16) JACAP_SELECT(32, 512);
  else if (max_seqlen <= 1024 * 4) JACAP_SELECT(4, 1024);
  else if (max_seqlen <= 1024 * 8) JACAP_SELECT(8, 1024);
  else if (max_seqlen <= 1024 * 16) JACAP_SELECT(16, 1024);
  else JACAP_SELECT(32, 1024);
#undef JACAP_SELECT
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
    JACAP_TRY(launch_pdl(dm.pdl != 0, compact_kernel<__nv_bfloat16>, blocks, 256, 0, st, dm, cu,
                         (const __nv_bfloat16*)k, (const __nv_bfloat16*)v, idx, budget, (__nv_bfloat16*)k_out,
                         (__nv_bfloat16*)v_out));
  else
    JACAP_TRY(launch_pdl(dm.pdl != 0, compact_kernel<float>, blocks, 256, 0, st, dm, cu, (const float*)k,
                         (const float*)v, idx, budget, (float*)k_out, (float*)v_out));
  return cudaGetLastError();
}

}  // namespace jacap
