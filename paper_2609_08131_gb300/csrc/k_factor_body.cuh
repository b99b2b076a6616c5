// k_factor_body.cuh - the blocked factor as a device function: the kernel
// of k_factor.cu and the factor role of the fused schedule (k_fused.cu)
// both run it. See k_factor.cu for what it computes.
#pragma once

#include "jacap_dev.cuh"

namespace jacap {

constexpr int FA_THREADS = 256;
constexpr int FA_ROWS = D * 32 / FA_THREADS;  // 16 rows per thread

// 1/p: approximate reciprocal refined by one Newton-Raphson step.
__device__ __forceinline__ float recip_nr(float p) {
  float x;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(x) : "f"(p));
  return x * fmaf(-p, x, 2.f);
}
// ------------------------------------------------------------ blocked ------
// The proxy path (u = v) factors A with a blocked right-looking Cholesky on
// 32 x 32 blocks (I, J = 0..3) and inverts the factor blockwise, so the
// sequential part is four 32-step eliminations inside one warp instead of
// 128 block-wide steps:
//  for K = 0..3:
//    T_KK = L_KK^{-1}   one warp: the forward elimination above on the 32 x 32
//                       block A_KK (its lower triangle), X_KK -> T_KK
//    L_IK = A_IK T_KK^T                 I > K
//    A_IJ -= L_IK L_JK^T                K < J <= I
//  X = L^{-1}:  X_II = T_II,  X_IJ = -T_II S_IJ,  S_IJ = sum_{M=J}^{I-1} L_IM X_MJ
//  (I > J). Phase P of the inverse (P = 0 .. 3) forms X_PJ = -T_PP S_PJ for
//  J < P and adds the terms M = P, S_IJ += L_IP X_PJ (I > P, J <= P); it needs
//  only blocks of step P and earlier, so phases 0-2 run on six warps while
//  warp 0 eliminates the next diagonal block, and only X_3J follows the last
//  elimination.
// Every product is a 32 x 32 block of "rows times rows" (P Q^T) read from
// shared memory with row stride FB_LD; the inverse is built transposed
// (XT_JI = X_IJ^T) so its products have that form too. Thread t owns the
// outputs (a + 16 p, b + 16 q), a = t / 16, b = t % 16, p, q in {0, 1}.
constexpr int FB_THREADS = 256;
constexpr int FB_LD = 36;             // row stride of a 32 x 32 block (floats); 16-byte rows
constexpr int FB_BLK = 32 * FB_LD;    // floats per block
// 10 lower blocks of A (then L_IJ, and T_II on the diagonal) and 10 blocks of
// XT (XT_JI at tri(I, J); S_IJ^T there until X_IJ replaces it)
// 10 lower blocks of A and 10 of XT, then the elimination's buffers (192 floats)
constexpr int FB_ELIM = 192;
constexpr size_t FB_SMEM = ((size_t)20 * FB_BLK + FB_ELIM) * sizeof(float);

__device__ __forceinline__ int tri(int i, int j) { return i * (i + 1) / 2 + j; }  // block (i, j), j <= i
// a partial Gram's lower blocks staged in shared memory: column block nb,
// rows 32 nb .. 127, 32 floats per row, after the segments of blocks < nb
__host__ __device__ constexpr int fb_seg(int nb) { return 32 * (128 * nb - 16 * nb * (nb - 1)); }
constexpr int FB_STAGE = fb_seg(4);  // floats per stage (10 blocks of 32 x 32)
static_assert(2 * FB_STAGE <= 20 * FB_BLK, "the staging ring fits in the A and XT blocks");
// partials in flight: 2 in the factor kernel (two CTAs per SM), 5 in the fused
// schedule's factor role (one CTA per SM, the shared memory of the Gram role)
template <bool FUSED> __host__ __device__ constexpr int fb_stages() { return FUSED ? 5 : 2; }
// floats before the elimination buffers: the A and XT blocks, or the staging ring if that is longer
template <bool FUSED> __host__ __device__ constexpr int fb_elim_at() {
  return 20 * FB_BLK > fb_stages<FUSED>() * FB_STAGE ? 20 * FB_BLK : fb_stages<FUSED>() * FB_STAGE;
}
static_assert(fb_elim_at<false>() == 20 * FB_BLK, "the factor kernel's shared memory");
constexpr size_t FB_FUSED_SMEM = ((size_t)fb_elim_at<true>() + FB_ELIM) * sizeof(float);

// The barrier of the factor's FB_THREADS threads (named barrier 1: in the
// fused schedule the factor runs on the first FB_THREADS threads of a larger CTA).
__device__ __forceinline__ void fb_all() { named_barrier_sync(1, FB_THREADS); }

// acc[p][q] += sum_m P[a + 16 p][m] Q[b + 16 q][m], with packed fp32x2
// multiply-adds: the even and the odd m accumulate separately and are added
// at the end (half the instructions of one chain per output)
__device__ __forceinline__ void nt_block(float (&acc)[2][2], const float* P, const float* Q, int a, int b) {
  float2 s[2][2];
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int j = 0; j < 2; ++j) s[i][j] = make_float2(0.f, 0.f);
#pragma unroll
  for (int m = 0; m < 32; m += 4) {
    const float4 p0 = *(const float4*)(P + a * FB_LD + m);
    const float4 p1 = *(const float4*)(P + (a + 16) * FB_LD + m);
    const float4 q0 = *(const float4*)(Q + b * FB_LD + m);
    const float4 q1 = *(const float4*)(Q + (b + 16) * FB_LD + m);
    const float4 pv[2] = {p0, p1}, qv[2] = {q0, q1};
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        s[i][j] = __ffma2_rn(make_float2(pv[i].x, pv[i].y), make_float2(qv[j].x, qv[j].y), s[i][j]);
        s[i][j] = __ffma2_rn(make_float2(pv[i].z, pv[i].w), make_float2(qv[j].z, qv[j].w), s[i][j]);
      }
  }
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int j = 0; j < 2; ++j) acc[i][j] += s[i][j].x + s[i][j].y;
}

// T = L^{-1} of one 32 x 32 diagonal block by the elimination described at the
// top of the file, in one warp: lane r holds row r in registers. At step k the
// pivot row goes to every lane through shared memory: its scaled inverse part
// (columns < k) from lane k's registers, its A part (columns >= k) as column k
// of every row (the lower triangle of A; each lane stores its own element).
// The steps are software-pipelined: step k first updates column k + 1 (the
// next pivot column), sends the next pivot p_{k+1} and row k + 2's element in
// column k + 1 by shuffle and starts their reciprocal, updates the inverse
// part, stores the next pivot row, and only then makes the rest of its
// multiply-adds, which hide the latency of the stores, the shuffles and the
// reciprocal; the next pivot row is loaded after them. rb, cb: two 32-float
// buffers each (16-byte aligned), alternating by step; piv, pinv: the 32
// pivots and their reciprocals. Writes T row-major into `blk` and T^T into
// `tblk`.
__device__ __forceinline__ void diag_inverse(float* blk, float* tblk, float* rb, float* cb, float* piv, float* pinv,
                                             int lane, bool& bad) {
  float z[32];
#pragma unroll
  for (int c = 0; c < 32; c += 4) {
    const float4 v = *(const float4*)(blk + lane * FB_LD + c);
    z[c] = v.x;
    z[c + 1] = v.y;
    z[c + 2] = v.z;
    z[c + 3] = v.w;
  }
  // step 0's pivot row is column 0 of every row (no inverse part yet)
  cb[lane] = z[0];
  float p = __shfl_sync(0xffffffffu, z[0], 0);
  float rn = __shfl_sync(0xffffffffu, z[0], 1);  // A_{1,0}
  float inv = recip_nr(p);
  if (lane == 0) {
    piv[0] = p;
    pinv[0] = inv;
  }
  __syncwarp();
  float r[32];
#pragma unroll
  for (int c = 0; c < 32; c += 4) {
    const float4 v = *(const float4*)(cb + c);
    r[c] = v.x, r[c + 1] = v.y, r[c + 2] = v.z, r[c + 3] = v.w;
  }
#pragma unroll
  for (int k = 0; k < 32; ++k) {
    const float m = lane > k ? z[k] * inv : 0.f;
    float inv_next = 0.f;
    if (k + 1 < 32) {
      z[k + 1] = fmaf(-m, rn, z[k + 1]);  // the next pivot column first
      p = __shfl_sync(0xffffffffu, z[k + 1], k + 1);
      rn = k + 2 < 32 ? __shfl_sync(0xffffffffu, z[k + 1], k + 2) : 0.f;  // A_{k+2,k+1}
    }
#pragma unroll
    for (int c = 0; c < k; ++c) z[c] = fmaf(-m, r[c], z[c]);  // the inverse part
    if (k + 1 < 32) {
      // the pivot row of step k + 1: lane k + 1's inverse part (its columns
      // <= k are final now) and column k + 1 of every row
      float* rk = rb + ((k + 1) & 1) * 32;
      float* ck = cb + ((k + 1) & 1) * 32;
      ck[lane] = z[k + 1];
      if (lane == k + 1) {
#pragma unroll
        for (int c = 0; c <= k; c += 4) *(float4*)(rk + c) = make_float4(z[c], z[c + 1], z[c + 2], z[c + 3]);
      }
      inv_next = recip_nr(p);
      if (lane == 0) {
        piv[k + 1] = p;
        pinv[k + 1] = inv_next;
      }
    }
#pragma unroll
    for (int c = k + 2; c < 32; ++c) z[c] = fmaf(-m, r[c], z[c]);
    if (k + 1 < 32) {
      __syncwarp();
      const float* rk = rb + ((k + 1) & 1) * 32;
      const float* ck = cb + ((k + 1) & 1) * 32;
      const int kn = k + 1;
#pragma unroll
      for (int c = 0; c < 32; c += 4) {
        if (c + 4 <= kn) {
          const float4 v = *(const float4*)(rk + c);
          r[c] = v.x, r[c + 1] = v.y, r[c + 2] = v.z, r[c + 3] = v.w;
        } else if (c >= kn) {
          const float4 v = *(const float4*)(ck + c);
          r[c] = v.x, r[c + 1] = v.y, r[c + 2] = v.z, r[c + 3] = v.w;
        } else {  // the group that holds column kn: inverse part below kn, A part from kn on
          const float4 u = *(const float4*)(rk + c), v = *(const float4*)(ck + c);
          const float uu[4] = {u.x, u.y, u.z, u.w}, vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
          for (int j = 0; j < 4; ++j) r[c + j] = c + j < kn ? uu[j] : vv[j];
        }
      }
      inv = inv_next;
    }
  }
  // T_rc = X_rc / sqrt(p_r), X_rc = -z_c / p_c (c < r), X_rr = 1; the final
  // rows go through shared memory so that few registers stay live
#pragma unroll
  for (int c = 0; c < 32; c += 4) *(float4*)(blk + lane * FB_LD + c) = make_float4(z[c], z[c + 1], z[c + 2], z[c + 3]);
  __syncwarp();
  const float pr = piv[lane];
  if (!(pr > 0.f) || !isfinite(pr)) bad = true;
  const float sc = rsqrtf(fmaxf(pr, 1e-30f));
#pragma unroll
  for (int c = 0; c < 32; c += 4) {
    const float4 zz = *(const float4*)(blk + lane * FB_LD + c);
    const float4 iv = *(const float4*)(pinv + c);
    const float zv[4] = {zz.x, zz.y, zz.z, zz.w}, ivv[4] = {iv.x, iv.y, iv.z, iv.w};
    float t[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float x = c + j < lane ? -zv[j] * ivv[j] : (c + j == lane ? 1.f : 0.f);
      t[j] = x * sc;
      if (!isfinite(t[j])) bad = true;
      tblk[(c + j) * FB_LD + lane] = t[j];
    }
    *(float4*)(blk + lane * FB_LD + c) = make_float4(t[0], t[1], t[2], t[3]);
  }
}

// The trailing update of block step K: block i of the pairs K < J <= I < 4 in
// the order (I, J) = (K+1, K+1), (K+2, K+1), (K+2, K+2), ...
__device__ __forceinline__ void trailing_pair(int K, int i, int& I, int& J) {
  I = K + 1;
  J = K + 1;
  for (int n = 0; n < i; ++n) {
    if (J < I) {
      ++J;
    } else {
      ++I;
      J = K + 1;
    }
  }
}

// A_IJ -= L_IK L_JK^T for the trailing pairs i0 .. i1 - 1 of step K, by
// `nthr` threads (thread index vt), each taking a thread's share of one block
__device__ __forceinline__ void trailing_update(float* As, int K, int i0, int i1, int vt, int nthr) {
  for (int w = vt; w < (i1 - i0) * FB_THREADS; w += nthr) {
    int I, J;
    trailing_pair(K, i0 + w / FB_THREADS, I, J);
    const int t = w % FB_THREADS, a = t >> 4, b = t & 15;
    float d[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
    nt_block(d, As + tri(I, K) * FB_BLK, As + tri(J, K) * FB_BLK, a, b);
    float* o = As + tri(I, J) * FB_BLK;
#pragma unroll
    for (int p = 0; p < 2; ++p)
#pragma unroll
      for (int q = 0; q < 2; ++q) o[(a + 16 * p) * FB_LD + b + 16 * q] -= d[p][q];
  }
}

// Threads vt = 0 .. nthr - 1 (nthr = 192 or 256) meet at barrier `bar` (0:
// the whole CTA).
__device__ __forceinline__ void fb_sync(int bar, int nthr) {
  if (bar == 0) fb_all();
  else named_barrier_sync(bar, nthr);
}

// Inverse phase P, first half: X_PJ = -T_PP S_PJ for J < P, in place over
// S_PJ^T (XT(tri(P, J))). At most three 32 x 32 blocks' thread shares per thread.
__device__ __forceinline__ void inv_rows(float* As, float* XT, int P, int vt, int nthr, int bar) {
  float acc[3][2][2];
  const int items = P * FB_THREADS;
#pragma unroll
  for (int q = 0; q < 3; ++q) {
    acc[q][0][0] = acc[q][0][1] = acc[q][1][0] = acc[q][1][1] = 0.f;
    const int w = vt + q * nthr;
    if (w < items) {
      const int J = w / FB_THREADS, t = w % FB_THREADS;
      nt_block(acc[q], XT + tri(P, J) * FB_BLK, As + tri(P, P) * FB_BLK, t >> 4, t & 15);  // (T S)^T
    }
  }
  fb_sync(bar, nthr);  // every S_PJ is read before any X_PJ overwrites it
#pragma unroll
  for (int q = 0; q < 3; ++q) {
    const int w = vt + q * nthr;
    if (w < items) {
      const int J = w / FB_THREADS, t = w % FB_THREADS, a = t >> 4, b = t & 15;
      float* X = XT + tri(P, J) * FB_BLK;
#pragma unroll
      for (int i = 0; i < 2; ++i)
#pragma unroll
        for (int j = 0; j < 2; ++j) X[(a + 16 * i) * FB_LD + b + 16 * j] = -acc[q][i][j];
    }
  }
  fb_sync(bar, nthr);
}

// Inverse phase P, second half: S_IJ += L_IP X_PJ for I > P, J <= P (X_PP =
// T_PP); the first term of S_IJ (P == J) overwrites.
__device__ __forceinline__ void inv_accumulate(float* As, float* XT, int P, int vt, int nthr) {
  const int nj = P + 1;
  for (int w = vt; w < (3 - P) * nj * FB_THREADS; w += nthr) {
    const int blk = w / FB_THREADS, t = w % FB_THREADS, a = t >> 4, b = t & 15;
    const int I = P + 1 + blk / nj, J = blk % nj;
    float d[2][2] = {{0.f, 0.f}, {0.f, 0.f}};
    nt_block(d, XT + tri(P, J) * FB_BLK, As + tri(I, P) * FB_BLK, a, b);  // (L_IP X_PJ)^T
    float* S = XT + tri(I, J) * FB_BLK;
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        float* e = S + (a + 16 * i) * FB_LD + b + 16 * j;
        *e = (J == P) ? d[i][j] : *e + d[i][j];
      }
  }
}

// Units first, first + stride, ... of the CTA, one after the other, by its
// first FB_THREADS threads (further threads of the CTA must not call this).
// FUSED: the role of the fused schedule (k_fused.cu): each unit waits until
// the Gram role has completed it (6 progress counts per chunk), reads the
// partials with the L2 evict_first policy, and is published (fdone) once
// G, L^{-1} and the image are visible device-wide.
template <bool FUSED>
__device__ __forceinline__ void factor_blocked_cta(const Dims& dm, const Ws& ws, int first, int stride) {
  extern __shared__ __align__(16) float fsm[];
  float* As = fsm;                // tri(I, J): A_IJ, then L_IJ (I > J) / T_II (I == J)
  float* XT = fsm + 10 * FB_BLK;  // tri(I, J): XT_JI = (L^{-1})_IJ^T
  constexpr int NST = fb_stages<FUSED>();
  __shared__ __align__(8) uint64_t s_full[NST];
  float* s_elim = fsm + fb_elim_at<FUSED>();  // the elimination's row and column buffers, pivots, reciprocals
  __shared__ int s_skip, s_bad, s_np;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    s_skip = status_failed(ws) ? 1 : 0;
    for (int i = 0; i < NST; ++i) mbar_init(smem_u32(&s_full[i]), 1);
    fence_mbar_init();
  }
  fb_all();
  if (s_skip) return;
  const int units = dm.L * dm.Hkv * dm.S;
  uint32_t kk = 0;  // partial stages consumed so far (phases of s_full across units)
  const uint64_t drop = FUSED ? policy_evict_first() : 0;
  // time accounting (trace builds, thread 0, the elimination warp): 0 the
  // partial Grams summed into A (and G stored), 1-4 the eliminations of the
  // diagonal blocks, 5 its waits for the other warps after them, 6 panels and
  // look-ahead updates, 7 the last inverse phase, 8 the outputs, 9 units,
  // 10 the whole unit
  TRC_DECL(TR_CTA_SLOTS);
#pragma unroll 1
  for (int u = first; u < units; u += stride) {
  TRC_T(tr_unit);
  TRC_INC(9);
  const int plane = u / dm.S, s = u % dm.S;
  const int ch0 = ws.plan[1 + s], ch1 = ws.plan[2 + s];
  const float* gp = ws.gpart + ((int64_t)plane * dm.c_cap) * D * D;
  bool bad = false;
  int unit_np = 0;  // partials of this unit
  if (tid == 0) s_bad = 0;

  // A = I + sum of the unit's partial Grams (chunk order) over the lower
  // 32 x 32 blocks (the partials hold only those); G to the workspace and the lower blocks of
  // A to shared memory. The partials stream through a two-stage ring of bulk
  // copies (the 4 lower segments of one partial per stage: rows 32 nb .. 127
  // of column block nb, contiguous in the partial layout) while the threads
  // add the previous stage. Thread (ty, tx) sums rows ty + 8 a, columns
  // 4 tx .. 4 tx + 3; rows ty + 8 a lie in block a / 4.
  float* gout = ws.gram + (int64_t)u * D * D;
  {
    // the chunks that hold partials (the first chunk of every run)
    const int32_t* pf = ws.pflag + (int64_t)plane * dm.c_cap;
    if (tid == 0) {
      int np = 0;
      if (FUSED) {  // every item of the unit has stored its weights and partial
        if (wait_count(ws.gcount + u, 6 * (ch1 - ch0), ws, nullptr)) fence_proxy_async_global();
        else np = -1;
        JACAP_TRACE_MAX(ws, u, TR_FAC0);
      }
      if (np == 0)
        for (int ch = ch0; ch < ch1; ++ch) np += pf[ch] != 0;
      s_np = np;
    }
    fb_all();
    const int np = s_np;
    if (np < 0) return;  // the pass failed elsewhere, or the wait ran out
    unit_np = np;
    int cursor = ch0;  // (thread 0) next chunk to look at for a partial
    auto next_partial = [&]() {
      while (cursor < ch1 && !pf[cursor]) ++cursor;
      return cursor++;
    };
    auto issue = [&](int ch, int st) {  // one partial into stage st
      uint8_t* dst = (uint8_t*)(fsm + st * FB_STAGE);
      const float* src = gp + (int64_t)ch * D * D;
      mbar_arrive_expect_tx(smem_u32(&s_full[st]), FB_STAGE * 4);
#pragma unroll
      for (int nb = 0; nb < 4; ++nb) {
        const uint32_t sd = smem_u32(dst + fb_seg(nb) * 4), bytes = (D - 32 * nb) * 32 * 4;
        const float* sp = src + (nb * D + 32 * nb) * 32;
        if (FUSED) bulk_g2s_hint(sd, sp, bytes, smem_u32(&s_full[st]), drop);
        else bulk_g2s(sd, sp, bytes, smem_u32(&s_full[st]));
      }
    };
    if (tid == 0) {
      fence_proxy_async_smem();  // the previous unit's generic writes to the staging area come first
      for (int k = 0; k < NST && k < np; ++k) issue(next_partial(), (kk + k) % NST);
    }
    const int ty = tid >> 5, tx = tid & 31, c0 = 4 * tx;
    const int J = c0 >> 5, c = c0 & 31;
    float4 z[FA_ROWS];
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a) z[a] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int k = 0; k < np; ++k) {
      const uint32_t kg = kk + k;
      const int st = kg % NST;
      if (!mbar_wait(smem_u32(&s_full[st]), (kg / NST) & 1, ws, nullptr)) bad = true;
      const float* sb = fsm + st * FB_STAGE + fb_seg(J) + c;
#pragma unroll
      for (int a = 0; a < FA_ROWS; ++a) {
        if (a / 4 < J) continue;  // upper block
        const float4 v = *(const float4*)(sb + (ty + 8 * a - 32 * J) * 32);
        z[a].x += v.x;
        z[a].y += v.y;
        z[a].z += v.z;
        z[a].w += v.w;
      }
      fb_all();  // stage st is read; it may be refilled
      if (tid == 0 && k + NST < np) {
        fence_proxy_async_smem();
        issue(next_partial(), st);
      }
    }
#pragma unroll
    for (int a = 0; a < FA_ROWS; ++a) {
      const int i = ty + 8 * a, I = a / 4;
      if (I < J) continue;
      *(float4*)(gout + i * D + c0) = z[a];
      float4 v = z[a];
      v.x += i == c0 ? 1.f : 0.f;
      v.y += i == c0 + 1 ? 1.f : 0.f;
      v.z += i == c0 + 2 ? 1.f : 0.f;
      v.w += i == c0 + 3 ? 1.f : 0.f;
      *(float4*)(As + tri(I, J) * FB_BLK + (i & 31) * FB_LD + c) = v;
    }
  }
  fb_all();
  // the upper blocks of G by symmetry: G_IJ = A_JI^T (I < J), 4 x 4 tiles
  // transposed in registers
  for (int e = tid; e < 6 * 64; e += FB_THREADS) {
    const int ub = e >> 6, si = e & 7, sj = (e >> 3) & 7;
    const int I = ub < 3 ? 0 : (ub < 5 ? 1 : 2), J = ub < 3 ? ub + 1 : (ub < 5 ? ub - 1 : 3);
    const float* src = As + tri(J, I) * FB_BLK + (4 * sj) * FB_LD + 4 * si;
    float4 r[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) r[k] = *(const float4*)(src + k * FB_LD);
    float* dst = gout + (32 * I + 4 * si) * D + 32 * J + 4 * sj;
    *(float4*)(dst) = make_float4(r[0].x, r[1].x, r[2].x, r[3].x);
    *(float4*)(dst + D) = make_float4(r[0].y, r[1].y, r[2].y, r[3].y);
    *(float4*)(dst + 2 * D) = make_float4(r[0].z, r[1].z, r[2].z, r[3].z);
    *(float4*)(dst + 3 * D) = make_float4(r[0].w, r[1].w, r[2].w, r[3].w);
  }

  TRC_ADD(0, tr_unit);
  const int a = tid >> 4, b = tid & 15;
  // the six warps off warp 0's sub-partition (1-3, 5-7) work next to the
  // elimination, so it keeps its issue slots
  const int vt = (warp < 4 ? warp - 1 : warp - 2) * 32 + lane;
  // Block step K: warp 0 eliminates the diagonal block A_KK while the six
  // warps finish step K-1's trailing update (all but its first pair, the
  // block A_KK itself, which was updated ahead) and run inverse phase K - 1;
  // then all warps form the panel L_IK and update the next diagonal block
  // A_{K+1,K+1} first, so the next elimination can start.
#pragma unroll 1
  for (int K = 0; K < 4; ++K) {
    if (warp == 0) {
      TRC_T(tr_e);
      diag_inverse(As + tri(K, K) * FB_BLK, XT + tri(K, K) * FB_BLK, s_elim, s_elim + 64, s_elim + 128, s_elim + 160,
                   lane, bad);
      TRC_ADD(1 + K, tr_e);
    } else if (warp != 4 && K >= 1) {
      trailing_update(As, K - 1, 1, (4 - K) * (5 - K) / 2, vt, 192);
      inv_rows(As, XT, K - 1, vt, 192, 2);
      inv_accumulate(As, XT, K - 1, vt, 192);
    }
    TRC_T(tr_w);
    fb_all();
    TRC_ADD(5, tr_w);
    TRC_T(tr_p);
    // L_IK = A_IK T_KK^T for I > K
    float acc[3][2][2];
#pragma unroll
    for (int q = 0; q < 3; ++q) {
      acc[q][0][0] = acc[q][0][1] = acc[q][1][0] = acc[q][1][1] = 0.f;
      if (K + 1 + q < 4) nt_block(acc[q], As + tri(K + 1 + q, K) * FB_BLK, As + tri(K, K) * FB_BLK, a, b);
    }
    fb_all();
#pragma unroll
    for (int q = 0; q < 3; ++q)
      if (K + 1 + q < 4) {
        float* L = As + tri(K + 1 + q, K) * FB_BLK;
#pragma unroll
        for (int i = 0; i < 2; ++i)
#pragma unroll
          for (int j = 0; j < 2; ++j) L[(a + 16 * i) * FB_LD + b + 16 * j] = acc[q][i][j];
      }
    fb_all();
    if (K == 3) {
      TRC_ADD(6, tr_p);
      break;
    }
    // A_{K+1,K+1} -= L_{K+1,K} L_{K+1,K}^T ahead of the rest of the trailing update
    trailing_update(As, K, 0, 1, tid, FB_THREADS);
    fb_all();
    TRC_ADD(6, tr_p);
  }

  // inverse phase 3: X_3J = -T_33 S_3J (all threads)
  TRC_T(tr_t);
  inv_rows(As, XT, 3, tid, FB_THREADS, 0);
  TRC_ADD(7, tr_t);
  TRC_T(tr_o);
  if (bad) s_bad = 1;

  // Outputs, 64 rows of L^{-1} at a time, staged row-major in the A blocks
  // (free now) so that every global store is a full 512-byte row (float32)
  // or a run of 128-byte image rows: L^{-1}[n][c] = XT(tri(n / 32, c / 32))
  // [c % 32][n % 32] for n >= c, 0 above. Reading XT with consecutive n per
  // warp and writing the padded staging rows are both free of bank conflicts
  // beyond the minimum.
  float* mout = ws.minv + (int64_t)u * D * D;
  uint8_t* img = ws.minv_img + (int64_t)u * 65536;
  constexpr int ST_LD = D + 4;
  float* stage = As;  // [64][ST_LD]
  static_assert(64 * ST_LD <= 10 * FB_BLK, "staging fits in the A blocks");
#pragma unroll 1
  for (int half = 0; half < 2; ++half) {
    {
      const int nl = tid & 63, cg = tid >> 6;  // row of the half, 32-column group
      const int n = 64 * half + nl;
      const float* src = XT + tri(n >> 5, cg) * FB_BLK + (n & 31);
#pragma unroll
      for (int j = 0; j < 32; j += 4) {
        float x[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int c = 32 * cg + j + q;
          x[q] = (cg <= (n >> 5) && c <= n) ? src[(j + q) * FB_LD] : 0.f;
        }
        *(float4*)(stage + nl * ST_LD + 32 * cg + j) = make_float4(x[0], x[1], x[2], x[3]);
      }
    }
    fb_all();
    // float32 rows: one 512-byte row per warp instruction
#pragma unroll
    for (int r = warp; r < 64; r += FB_THREADS / 32)
      *(float4*)(mout + (64 * half + r) * D + 4 * lane) = *(const float4*)(stage + r * ST_LD + 4 * lane);
    // bf16 hi/lo image: 2 K-atoms (channels 0-63, 64-127) x 256 rows x 128 B;
    // lanes 8 a .. 8 a + 7 take the eight 16-byte chunks of one atom row
#pragma unroll 1
    for (int e = tid; e < 64 * 16; e += FB_THREADS) {
      const int nl = e >> 4, at = (e >> 3) & 1, ch = e & 7;
      const int n = 64 * half + nl;
      const float4 x0 = *(const float4*)(stage + nl * ST_LD + 64 * at + 8 * ch);
      const float4 x1 = *(const float4*)(stage + nl * ST_LD + 64 * at + 8 * ch + 4);
      const float x[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
      uint32_t hi[4], lo[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        hi[q] = pack_bf16x2(x[2 * q], x[2 * q + 1]);
        lo[q] = pack_bf16x2(x[2 * q] - bf16lo(hi[q]), x[2 * q + 1] - bf16hi(hi[q]));
      }
      // hi and lo of row n at image rows 32 (n / 16) + n % 16 and 16 further
      const uint32_t ir = 32 * (n >> 4) + (n & 15);
      *(uint4*)(img + at * 32768 + sw128_off(ir, ch)) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
      *(uint4*)(img + at * 32768 + sw128_off(ir + 16, ch)) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    }
    fb_all();
  }
  kk += (uint32_t)unit_np;
  if (tid == 0 && s_bad) flag(ws, ST_NONFINITE);
  if (FUSED) {  // G, L^{-1} and the image are visible device-wide: publish the unit
    fence_proxy_async_global();
    __threadfence();
    fb_all();
    if (tid == 0) {
      st_release_gpu(ws.fdone + u, 1);
      JACAP_TRACE_MAX(ws, u, TR_FAC1);
    }
  }
  TRC_ADD(8, tr_o);
  TRC_ADD(10, tr_unit);
  }
  if (tid == 0) TRC_PUT(ws, TR_K_FACTOR, 11);
}

}  // namespace jacap
