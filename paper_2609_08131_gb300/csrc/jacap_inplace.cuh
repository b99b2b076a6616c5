// jacap_inplace.cuh - in-place compaction of one unit's kept rows, shared by
// the stand-alone compaction kernels (k_decode.cu) and the selection kernel
// that compacts each unit right after selecting it (k_select.cu). All NT
// threads of the CTA call these together; the kept positions ix[0 .. kept)
// ascend strictly within [0, n) (checked by the caller where they come from
// outside).
#pragma once

#include "jacap_dev.cuh"

namespace jacap {

constexpr int CI_CHUNK_BYTES = 16384;  // per tensor and chunk

// Ascending order: row r receives row ix[r]. Rows move in chunks that are
// read whole (a barrier) before any of them is written; since ix[r] >= r, a
// chunk's writes never touch a row that a later chunk still has to read.
template <typename T, int NT>
__device__ __forceinline__ void compact_ordered_unit(const Dims& dm, int plane, int64_t t0, int kept, T* k, T* v,
                                                     int32_t* pos, const int32_t* ix) {
  constexpr int RB = D * (int)sizeof(T) / 16;  // 16-byte pieces per row
  constexpr int CH = CI_CHUNK_BYTES / (D * (int)sizeof(T));
  constexpr int PER = CH * RB / NT;            // pieces per thread and tensor
  static_assert(CH * RB % NT == 0 && CH <= NT, "chunk shape");
  const int tid = threadIdx.x;
  const int l = plane / dm.Hkv, g = plane % dm.Hkv;
  const int64_t rowoff = (int64_t)l * dm.kv_sl + (int64_t)g * dm.kv_sh;
  uint4* kb = (uint4*)(k + rowoff);
  uint4* vb = (uint4*)(v + rowoff);
  const int64_t st16 = dm.kv_st * (int64_t)sizeof(T) / 16;  // token stride in 16-byte pieces
  // the tags follow the layout of K with one int32 per token row
  int32_t* pb = pos != nullptr ? pos + (int64_t)l * (dm.kv_sl / dm.kv_st) + (int64_t)g * (dm.kv_sh / dm.kv_st) : nullptr;
  for (int c0 = 0; c0 < kept; c0 += CH) {
    uint4 kr[PER], vr[PER];
    int32_t pr = 0;
#pragma unroll
    for (int e = 0; e < PER; ++e) {
      const int q = e * NT + tid, r = c0 + q / RB, piece = q % RB;
      if (r < kept) {
        const int32_t x = ix[r];
        if (x != r) {
          kr[e] = kb[(t0 + x) * st16 + piece];
          vr[e] = vb[(t0 + x) * st16 + piece];
        }
      }
    }
    if (pb != nullptr && tid < CH && c0 + tid < kept) pr = pb[t0 + ix[c0 + tid]];
    __syncthreads();  // the whole chunk is read before any of it is written
#pragma unroll
    for (int e = 0; e < PER; ++e) {
      const int q = e * NT + tid, r = c0 + q / RB, piece = q % RB;
      if (r < kept && ix[r] != r) {
        kb[(t0 + r) * st16 + piece] = kr[e];
        vb[(t0 + r) * st16 + piece] = vr[e];
      }
    }
    if (pb != nullptr && tid < CH && c0 + tid < kept) pb[t0 + c0 + tid] = pr;
  }
}

// Hole filling, given f = the number of kept positions below `kept`: the
// kept rows at or above `kept` move, in ascending order, into the evicted rows
// below `kept`. c(p) = ix[p] - p counts the evicted rows below kept position p
// and does not decrease, so hole j lies after the i = #{p < f : c(p) <= j}
// kept positions below it, at row j + i. One warp per hole (lanes over the
// 16-byte pieces of the row); sources and destinations are disjoint.
template <typename T, int NT>
__device__ __forceinline__ void fill_holes_unit(const Dims& dm, int plane, int64_t t0, int kept, int f, T* k, T* v,
                                                int32_t* pos, const int32_t* ix) {
  constexpr int RB = D * (int)sizeof(T) / 16;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int holes = kept - f;
  const int l = plane / dm.Hkv, g = plane % dm.Hkv;
  const int64_t rowoff = (int64_t)l * dm.kv_sl + (int64_t)g * dm.kv_sh;
  uint4* kb = (uint4*)(k + rowoff);
  uint4* vb = (uint4*)(v + rowoff);
  const int64_t st16 = dm.kv_st * (int64_t)sizeof(T) / 16;
  // the tags follow the layout of K with one int32 per token row
  int32_t* pb = pos != nullptr ? pos + (int64_t)l * (dm.kv_sl / dm.kv_st) + (int64_t)g * (dm.kv_sh / dm.kv_st) : nullptr;
  for (int j = warp; j < holes; j += NT / 32) {
    int lo = 0, hi = f;  // first p in [0, f) with c(p) > j (f if none)
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (ix[mid] - mid <= j) lo = mid + 1; else hi = mid;
    }
    const int64_t dst = t0 + j + lo, src = t0 + ix[f + j];
    for (int piece = lane; piece < RB; piece += 32) {
      kb[dst * st16 + piece] = kb[src * st16 + piece];
      vb[dst * st16 + piece] = vb[src * st16 + piece];
    }
    if (pb != nullptr && lane == 0) pb[dst] = pb[src];
  }
}

}  // namespace jacap
