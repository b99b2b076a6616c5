// jacap_dev.cuh - shared definitions of the libjacap kernels (sm_103a).
//
// Problem shapes, the workspace map, the work-item plan, and thin inline-PTX
// wrappers for mbarriers, TMA (cp.async.bulk.tensor), bulk copies and the
// tcgen05 tensor-core / tensor-memory instructions. Every wait on an mbarrier
// is bounded by wall-clock time (%globaltimer); on expiry the waiter records
// JACAP status bit ST_TIMEOUT in the workspace status word and reports failure
// to its caller, which then winds the CTA down instead of spinning forever.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace jacap {

constexpr int D = 128;     // head_dim d_k = d_o
constexpr int TILE = 128;  // tokens per tile (one TMA box row count, one MMA M)

// Status word bits (word 0 of the workspace). Host maps them to jacap_status.
enum : uint32_t {
  ST_INVALID = 1u,    // malformed cu_seqlens
  ST_NONFINITE = 2u,  // NaN/Inf in an input or intermediate
  ST_TIMEOUT = 4u,    // a bounded wait expired
};

constexpr unsigned long long WAIT_LIMIT_NS = 2000000000ull;  // 2 s per wait

// Shapes and method constants of one call, passed by value to every kernel.
struct Dims {
  int S, L, Hq, Hkv, G, window;
  int64_t Ntot;
  int chunk;          // tokens per work item (multiple of TILE)
  int64_t c_cap;      // capacity of per-plane chunk arrays (>= sum_s ceil(n_s/chunk))
  int64_t kv_sl, kv_sh, kv_st;  // K/V strides (elements)
  int64_t q_ss, q_sl, q_sh, q_sp;
  float inv_scale;    // 1 / (tau sqrt(d))
  float wdiv;         // 1/d (Eq. 8) or 1 (weight_div_dk = 0)
  int cov_unbiased;
  int linear;         // 1: S_C = I, rho = 1 (linear surrogate weight)
  int dense_minv;     // 1: the score matrix is a full 128 x 128 (output directions), not triangular
  int full_cov;       // 1: kappa with the full window covariance of the queries (App. B.2)
  int kf_rp;          // full covariance on the tensor cores: rows per split part of the query image (else 0)
  int pdl;            // 1: launch with programmatic stream serialization (0 when timing events sit between kernels)
  int fused;          // 1: the Gram, the factor and the scores run as roles of one persistent launch (k_fused.cu)
  int keep_tiles;     // fused: V tiles of each Gram item loaded with the L2 evict_last policy (the score
                      // role reads them again soon after); the item's other tiles are loaded evict_first
  int run_items;      // fused: consecutive items a role's CTA takes at a time (one partial Gram per run)
};

// Rows per split part of the full-covariance query image of one KV head's
// group (G heads x W window queries, padded to 32, 64 or 128 rows); 0 where
// the tensor-core kernel does not apply (window not in {8, 16, 32, 64} or more
// than 128 centred queries per group).
__host__ __device__ constexpr int kfull_rows_padded(int G, int W) {
  return (W == 8 || W == 16 || W == 32 || W == 64) && G * W <= 128 ? (G * W <= 32 ? 32 : (G * W <= 64 ? 64 : 128))
                                                                    : 0;
}

// Workspace map (device pointers into the caller's workspace).
struct Ws {
  uint32_t* status;   // [16] status word + first failing unit
  int32_t* plan;      // [0] = chunks per plane C_tot, [1 .. S+1] = chunk prefix per request
  int4* chunks;       // [c_cap] chunk r of every plane: {t0, t1, request, r}
  int32_t* gcount;    // [units] fused schedule: Gram progress of a unit (each item adds 1 for its weights
                      // and 1 for its partial Gram; complete at 2 x the unit's chunk count)
  int32_t* fdone;     // [units] fused schedule: 1 once the unit's factor (G, L^{-1} and its image) is written
  float* mu;          // [S][L][Hq][D]  mu / (tau sqrt d)
  float* lam;         // [S][L][Hq][D]  diagonal of Lambda_Q
  float* qdev;        // [S][L][Hq][window][D]  centred window queries q_j - mu (full covariance, CUDA cores)
  uint8_t* qimg;      // [S][L][Hkv][512 kf_rp]  the same as a bf16 hi/lo shared-memory image (tensor cores);
                      // shares qdev's section
  float* lk;          // [L*Hkv][Ntot][2G]  logits then kappa per query head of the group
  float* cstats;      // [L*Hkv][c_cap][G][2]  per-chunk (max, sum exp(l - max))
  float* ustats;      // [units][G][2]  the unit's softmax normaliser per head: (M_h, 1 / Z_h)
  float* w;           // [L*Hkv][Ntot]  Eq. 8 weights summed over the group
  float* gpart;       // [L*Hkv][c_cap][D/32][D][32]  partial Grams: (m, n) at ((n/32) D + m) 32 + n%32,
                      // lower 32 x 32 blocks only; one per run of a CTA's consecutive chunks of a unit,
                      // stored at the run's first chunk
  int32_t* pflag;     // [L*Hkv][c_cap]  1 where gpart holds a partial (a run's first chunk), else 0
  float* gram;        // [units][D][D]  sum_i w_i v_i v_i^T
  float* minv;        // [units][D][D]  L^{-1} (float32, lower triangular)
  uint8_t* minv_img;  // [units][65536]  L^{-1} as bf16 hi/lo, shared-memory image for the score MMA
  unsigned long long* trace;  // [units][8] timeline of the fused schedule (JACAP_TRACE builds only, else null)
  unsigned long long* trace_cta;  // [TR_KERNELS][TR_CTAS][TR_CTA_SLOTS] per-CTA time accounting (JACAP_TRACE)
};

// Timeline of the fused schedule, per unit (JACAP_TRACE builds; %globaltimer
// ns): slot 0 first Gram tile issued (min), 1 last Gram partial published
// (max), 2 factor start (its wait done), 3 factor published, 4 first score
// image acquired (min), 5 last score tile finished (max), 6 first score MMA
// issued (min). The plan kernel resets the slots.
enum { TR_GRAM0 = 0, TR_GRAM1, TR_FAC0, TR_FAC1, TR_SC_IMG, TR_SC1, TR_SC_MMA, TR_SLOTS = 8 };
// Per-CTA time accounting of the streaming kernels (JACAP_TRACE builds): for
// kernel k (TR_K_*) and CTA b, slot j of trace_cta[(k TR_CTAS + b) TR_CTA_SLOTS]
// sums the ns one role's lane 0 spent in a wait or a busy section (the slot
// meanings are listed where each kernel records them).
enum { TR_K_GRAM = 0, TR_K_SCORE = 1, TR_K_KPASS = 2, TR_K_FACTOR = 3, TR_K_SELECT = 4, TR_KERNELS = 5, TR_CTAS = 1024,
       TR_CTA_SLOTS = 16 };

// A unit is (plane p = l*Hkv + g, request s); its index is p*S + s.
struct Item {
  int plane, seq;         // plane and request
  int64_t t0, t1;         // token range [t0, t1) on the plane's token axis
  int cidx;               // chunk index within the plane
};

// The work items of a persistent CTA: items start, start + stride, ... where
// item i = plane * C_tot + r is chunk r of the plane (chunks never straddle
// requests; the chunk table is the same for every plane). The record of the
// next item is loaded while the current one is processed, so an item
// boundary costs no dependent global loads.
struct ItemStream {
  // CTA `part` of `parts` walks the contiguous item range [part T / parts,
  // (part + 1) T / parts) of the T = L Hkv C_tot items (plane-major, chunks of
  // a plane in request order), so the counts differ by at most one item and
  // consecutive items mostly belong to one unit (accumulators and images
  // carry over between them).
  const int4* tab;
  int64_t i, end;
  int ctot;
  int4 rec;
#ifdef JACAP_CHECKED
  int64_t ntot;
  int nseq, nplanes;
  uint32_t* status;
#endif
  // Strided (the fused schedule): the items are cut into runs of R =
  // dm.run_items consecutive items and CTA `part` of `parts` walks runs part,
  // part + parts, ..., so the CTAs of a role sweep the units in order together
  // and each unit's items finish close in time.
  int64_t run_end, skip, runlen;
  __device__ __forceinline__ ItemStream(const Dims& dm, const Ws& ws, int64_t part, int64_t parts,
                                        bool strided = false)
      : tab(ws.chunks) {
#ifdef JACAP_CHECKED
    ntot = dm.Ntot;
    nseq = dm.S;
    nplanes = dm.L * dm.Hkv;
    status = ws.status;
#endif
    ctot = ws.plan[0];
    const int64_t total = (int64_t)dm.L * dm.Hkv * ctot;
    if (strided) {
      const int64_t R = dm.run_items > 0 ? dm.run_items : 1;
      i = part * R;
      run_end = i + R;
      skip = (parts - 1) * R;
      runlen = R;
      end = total;
    } else {
      i = part * total / parts;
      end = (part + 1) * total / parts;
      run_end = end;
      skip = 0;
      runlen = 0;
    }
    if (i < end) rec = tab[i % ctot];
  }
  __device__ __forceinline__ bool next(Item& it) {
    if (i >= end) return false;
    it.plane = (int)(i / ctot);
    it.t0 = rec.x;
    it.t1 = rec.y;
    it.seq = rec.z;
    it.cidx = rec.w;
#ifdef JACAP_CHECKED
    // checked build: a record outside the cache ends this CTA's items and is
    // reported (ST_INVALID) instead of being streamed
    if (it.t0 < 0 || it.t1 <= it.t0 || it.t1 > ntot || it.seq < 0 || it.seq >= nseq || it.cidx < 0 ||
        it.cidx >= ctot || it.plane >= nplanes) {
      atomicOr(status, 1u);
      i = end;
      return false;
    }
#endif
    if (++i == run_end) {
      i += skip;
      run_end = i + runlen;
    }
    if (i < end) rec = tab[i % ctot];
    return true;
  }
  // whether this CTA's next item exists and belongs to the same unit as `cur`
  // (the item last returned by next())
  __device__ __forceinline__ bool next_same_unit(const Item& cur) const {
    return i < end && (int)(i / ctot) == cur.plane && rec.z == cur.seq;
  }
};

// Largest GQA group (query heads per KV head) the kernels are compiled for.
constexpr int G_MAX = 8;

// The logits/kappa rows hold 2G floats per token: l_h at [0, G), kappa_h at
// [G, 2G). A row starts on a multiple of 2G floats from a 1 KB-aligned base, so
// it is 16-byte aligned for even G and 8-byte aligned for odd G; the kappa
// half (G floats further) keeps 16 bytes only when G % 4 == 0.
template <int G>
struct LkAlign {
  static constexpr int ROW = G % 2 == 0 ? 4 : 2;                      // floats
  static constexpr int KAPPA = G % 4 == 0 ? 4 : (G % 2 == 0 ? 2 : 1);  // floats
};

// dst[0 .. N) = v with the widest stores an alignment of A floats (1, 2 or 4)
// allows.
template <int N, int A>
__device__ __forceinline__ void store_floats(float* dst, const float* v) {
  int e = 0;
  if constexpr (A >= 4) {
#pragma unroll
    for (; e + 4 <= N; e += 4) *(float4*)(dst + e) = make_float4(v[e], v[e + 1], v[e + 2], v[e + 3]);
  }
  if constexpr (A >= 2) {
#pragma unroll
    for (; e + 2 <= N; e += 2) *(float2*)(dst + e) = make_float2(v[e], v[e + 1]);
  }
#pragma unroll
  for (; e < N; ++e) dst[e] = v[e];
}

// v[0 .. N) = src[0 .. N) with the widest loads an alignment of A floats allows.
template <int N, int A>
__device__ __forceinline__ void load_floats(float* v, const float* src) {
  int e = 0;
  if constexpr (A >= 4) {
#pragma unroll
    for (; e + 4 <= N; e += 4) {
      const float4 x = *(const float4*)(src + e);
      v[e] = x.x;
      v[e + 1] = x.y;
      v[e + 2] = x.z;
      v[e + 3] = x.w;
    }
  }
  if constexpr (A >= 2) {
#pragma unroll
    for (; e + 2 <= N; e += 2) {
      const float2 x = *(const float2*)(src + e);
      v[e] = x.x;
      v[e + 1] = x.y;
    }
  }
#pragma unroll
  for (; e < N; ++e) v[e] = src[e];
}

// Programmatic dependent launch. A kernel launched with the programmatic
// stream-serialization attribute is set up while the previous kernel of the
// stream still runs and is scheduled as its CTAs exit (no kernel here triggers
// its dependents early: measured, an early trigger made the pass slower). Every
// kernel starts with pdl_wait(), which blocks until the previous kernel has
// completed with its memory visible (a no-op for a normal launch). Nothing
// before pdl_wait() may touch global memory.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ bool status_failed(const Ws& ws) {
  return *((volatile uint32_t*)ws.status) != 0u;
}

__device__ __forceinline__ void flag(const Ws& ws, uint32_t bit) { atomicOr(ws.status, bit); }

// Merge two online-softmax partials (max m, sum s of exp(x - m)); m = -inf
// marks an empty partial.
__device__ __forceinline__ void softmax_merge(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  if (M == -INFINITY) return;
  s = (m == -INFINITY ? 0.f : s * expf(m - M)) + (m2 == -INFINITY ? 0.f : s2 * expf(m2 - M));
  m = M;
}

// Butterfly merge of (m, s) over the 32 lanes of a warp; every lane ends with
// the warp total (same value on every lane, fixed order: deterministic).
__device__ __forceinline__ void softmax_warp_merge(float& m, float& s) {
#pragma unroll
  for (int off = 16; off >= 1; off >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, off);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, off);
    softmax_merge(m, s, m2, s2);
  }
}

// ------------------------------------------------------------------ PTX ----
// Named barrier `id` over `count` threads (a multiple of 32).
__device__ __forceinline__ void named_barrier_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Named barrier that also ORs `pred` over its `count` threads: every thread
// gets the same answer, so a group can take one decision (say, to leave on
// abort) where a flag read by each thread after the barrier could differ
// between its threads and strand some at the next barrier.
__device__ __forceinline__ bool named_barrier_any(int id, int count, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)pred), "r"(id), "r"(count)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

#ifdef JACAP_TRACE
__device__ __forceinline__ void trace_min(const Ws& ws, int64_t u, int slot) {
  if (ws.trace != nullptr) atomicMin(ws.trace + u * TR_SLOTS + slot, globaltimer());
}
__device__ __forceinline__ void trace_max(const Ws& ws, int64_t u, int slot) {
  if (ws.trace != nullptr) atomicMax(ws.trace + u * TR_SLOTS + slot, globaltimer());
}
#define JACAP_TRACE_MIN(ws, u, slot) trace_min(ws, u, slot)
#define JACAP_TRACE_MAX(ws, u, slot) trace_max(ws, u, slot)
// time accounting: TRC_T(v) starts a stopwatch, TRC_ADD(acc, v) adds its
// elapsed ns to acc, TRC_PUT(ws, k, slot, acc) adds acc to the CTA's slot
#define TRC_DECL(n) unsigned long long trc[n] = {}
#define TRC_T(v) const unsigned long long v = globaltimer()
#define TRC_ADD(i, v) (trc[i] += globaltimer() - (v))
#define TRC_INC(i) (++trc[i])
#define TRC_PUT(ws, k, n)                                                                                \
  do {                                                                                                 \
    if ((ws).trace_cta != nullptr && blockIdx.x < TR_CTAS)                                             \
      for (int trc_j = 0; trc_j < (n); ++trc_j)                                                        \
        if (trc[trc_j])                                                                                \
          atomicAdd((ws).trace_cta + ((size_t)(k) * TR_CTAS + blockIdx.x) * TR_CTA_SLOTS + trc_j, trc[trc_j]); \
  } while (0)
#else
#define JACAP_TRACE_MIN(ws, u, slot) ((void)0)
#define JACAP_TRACE_MAX(ws, u, slot) ((void)0)
#define TRC_DECL(n) ((void)0)
#define TRC_T(v) ((void)0)
#define TRC_ADD(i, v) ((void)0)
#define TRC_INC(i) ((void)0)
#define TRC_PUT(ws, k, n) ((void)0)
#endif

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.release.cta.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Same test, but a thread whose phase is not complete may be suspended for up
// to `hint_ns` (it resumes as soon as the phase completes), so waiting warps
// stop competing for issue slots and shared-memory bandwidth.
__device__ __forceinline__ bool mbar_try_wait_suspend(uint32_t bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

constexpr uint32_t WAIT_SUSPEND_NS = 1000;

// Bounded wait for the phase with the given parity to complete. Returns false
// (after flagging ST_TIMEOUT) if it did not complete within limit_ns
// (WAIT_LIMIT_NS for every wait of the pass), or if *abort became nonzero
// while waiting.
static __device__ __noinline__ bool mbar_wait_slow(uint32_t bar, uint32_t parity, const Ws& ws,
                                            volatile int* abort, unsigned long long limit_ns = WAIT_LIMIT_NS) {
  if (abort != nullptr && *abort) return false;
  const unsigned long long t0 = globaltimer();
  for (uint32_t it = 0;; ++it) {
    if (mbar_try_wait_suspend(bar, parity, WAIT_SUSPEND_NS)) return true;
    if ((it & 7u) == 7u) {
      if (abort != nullptr && *abort) return false;
      if (globaltimer() - t0 > limit_ns) {
        flag(ws, ST_TIMEOUT);
        if (abort != nullptr) *abort = 1;
        return false;
      }
    }
  }
}

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, const Ws& ws,
                                          volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  return mbar_wait_slow(bar, parity, ws, abort);
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// 4-D tiled TMA load into shared memory, completion counted on `bar`.
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* map, int c0, int c1, int c2,
                                            int c3, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cta.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
      "l"(map), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
      : "memory");
}

// Linear bulk copy global -> shared (16-byte aligned, size multiple of 16).
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// L2 eviction-priority policies for the .L2::cache_hint forms of the copies
// below (per instruction; no device-wide L2 setting is touched).
__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// tma_load_4d with an L2 cache policy.
__device__ __forceinline__ void tma_load_4d_hint(uint32_t dst, const CUtensorMap* map, int c0, int c1, int c2,
                                                 int c3, uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cta.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(dst),
      "l"(map), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar), "l"(policy)
      : "memory");
}

// bulk_g2s with an L2 cache policy.
__device__ __forceinline__ void bulk_g2s_hint(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar,
                                              uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(policy)
      : "memory");
}

// Cross-CTA progress flags of the fused schedule. A producer's threads store
// their results, each makes them visible device-wide (__threadfence), the
// producers meet at a barrier, and one of them adds to (or sets) the flag with
// release semantics; a consumer reads the flag with acquire semantics. Data
// that the consumer then reads with bulk copies (the async proxy) is ordered
// after the acquire by fence_proxy_async_global.
__device__ __forceinline__ int ld_acquire_gpu(const int32_t* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_add_release_gpu(int32_t* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void st_release_gpu(int32_t* p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Bounded wait until *p >= target (acquire). Gives up, returning false, when
// the pass has failed elsewhere (status word set), when *abort is set, or
// after WAIT_LIMIT_NS (then it records ST_TIMEOUT and sets *abort).
static __device__ __noinline__ bool wait_count(const int32_t* p, int target, const Ws& ws, volatile int* abort) {
  if (ld_acquire_gpu(p) >= target) return true;
  const unsigned long long t0 = globaltimer();
  for (uint32_t it = 0;; ++it) {
    __nanosleep(128);
    if (ld_acquire_gpu(p) >= target) return true;
    if ((it & 15u) == 15u) {
      if ((abort != nullptr && *abort) || status_failed(ws)) return false;
      if (globaltimer() - t0 > WAIT_LIMIT_NS) {
        flag(ws, ST_TIMEOUT);
        if (abort != nullptr) *abort = 1;
        return false;
      }
    }
  }
}

__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(map) : "memory");
}

// ------------------------------------------------------------ tcgen05 ----
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem desc] * B[smem desc], kind::f16 (bf16 inputs, f32 accumulate).
__device__ __forceinline__ void umma_f16_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem desc], kind::f16. A (M x K) lives in tensor
// memory: lane = row, each 32-bit column packs two consecutive K elements.
__device__ __forceinline__ void umma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Four 8x8 b16 matrices from shared memory, transposed: lane l gives the
// address of row l % 8 of matrix l / 8; thread t receives, per matrix, rows
// 2 (t % 4) and 2 (t % 4) + 1 of column t / 4 packed (lower row in the low half).
__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                              uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

// Store to tensor memory, shape 16 lanes x 128 bits: thread t writes r0 to
// (lane t/4, column t%4) and r1 to (lane 8 + t/4, column t%4), relative to taddr.
__device__ __forceinline__ void tmem_st_16x128b(uint32_t taddr, uint32_t r0, uint32_t r1) {
  asm volatile("tcgen05.st.sync.aligned.16x128b.x1.b32 [%0], {%1, %2};" ::"r"(taddr), "r"(r0), "r"(r1)
               : "memory");
}

// Eight repetitions of the 16x128b store along columns: registers 2j, 2j+1
// go to columns 4j .. 4j + 3 (32 columns in all).
__device__ __forceinline__ void tmem_st_16x128b_x8(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.16x128b.x8.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// Store 16 consecutive 32-bit columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_st_32x32b_x16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

// Store 32 consecutive 32-bit columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_st_32x32b_x32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
      "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Arrive on `bar` once every tcgen05 op issued so far by this thread completed.
__device__ __forceinline__ void umma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
               : "memory");
}

// Load 32 consecutive f32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float* v) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
        "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
        "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Load two runs of 32 consecutive 32-bit columns of this thread's TMEM lane
// (at ta and tb) and wait for both: one asm statement, so no use of the
// registers can be scheduled before the wait.
__device__ __forceinline__ void tmem_ld32x2(uint32_t ta, uint32_t tb, uint32_t* a, uint32_t* b) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%64];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
      "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63}, [%65];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(a[0]), "=r"(a[1]), "=r"(a[2]), "=r"(a[3]), "=r"(a[4]), "=r"(a[5]), "=r"(a[6]), "=r"(a[7]),
        "=r"(a[8]), "=r"(a[9]), "=r"(a[10]), "=r"(a[11]), "=r"(a[12]), "=r"(a[13]), "=r"(a[14]), "=r"(a[15]),
        "=r"(a[16]), "=r"(a[17]), "=r"(a[18]), "=r"(a[19]), "=r"(a[20]), "=r"(a[21]), "=r"(a[22]), "=r"(a[23]),
        "=r"(a[24]), "=r"(a[25]), "=r"(a[26]), "=r"(a[27]), "=r"(a[28]), "=r"(a[29]), "=r"(a[30]), "=r"(a[31]),
        "=r"(b[0]), "=r"(b[1]), "=r"(b[2]), "=r"(b[3]), "=r"(b[4]), "=r"(b[5]), "=r"(b[6]), "=r"(b[7]),
        "=r"(b[8]), "=r"(b[9]), "=r"(b[10]), "=r"(b[11]), "=r"(b[12]), "=r"(b[13]), "=r"(b[14]), "=r"(b[15]),
        "=r"(b[16]), "=r"(b[17]), "=r"(b[18]), "=r"(b[19]), "=r"(b[20]), "=r"(b[21]), "=r"(b[22]), "=r"(b[23]),
        "=r"(b[24]), "=r"(b[25]), "=r"(b[26]), "=r"(b[27]), "=r"(b[28]), "=r"(b[29]), "=r"(b[30]), "=r"(b[31])
      : "r"(ta), "r"(tb)
      : "memory");
}

// Load 16 consecutive f32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor (tcgen05 format): start address, leading-
// and stride-dimension byte offsets, version 1, 128-byte swizzle.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;  // descriptor version for tcgen05
  d |= (uint64_t)2 << 61;  // 128-byte swizzle
  return d;
}

// Instruction descriptor of kind::f16: bf16 A and B, f32 D, dense.
// a_mn / b_mn: 1 if that operand is MN-major (transposed), 0 if K-major.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N, int a_mn, int b_mn) {
  return (1u << 4)                      // D format f32
         | (1u << 7)                    // A format bf16
         | (1u << 10)                   // B format bf16
         | ((uint32_t)a_mn << 15)       // A major
         | ((uint32_t)b_mn << 16)       // B major
         | ((uint32_t)(N >> 3) << 17)   // N / 8
         | ((uint32_t)(M >> 4) << 24);  // M / 16
}

// Byte offset of element (row, col) in a [rows][64]-element bf16 block stored
// with the 128-byte swizzle (the layout TMA writes for a {64, rows} box).
__device__ __forceinline__ uint32_t sw128_off(uint32_t row, uint32_t chunk16) {
  return row * 128u + ((chunk16 ^ (row & 7u)) << 4);
}

__device__ __forceinline__ float bf16lo(uint32_t x) { return __uint_as_float(x << 16); }
__device__ __forceinline__ float bf16hi(uint32_t x) { return __uint_as_float(x & 0xFFFF0000u); }

// Round two floats to bf16 (nearest even) and pack (a in the low half).
__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(b), "f"(a));
  return r;
}

// Explicit shared-memory loads from 32-bit shared addresses (the aligned views
// of the dynamic shared buffer are plain pointers to the compiler, which would
// otherwise emit generic loads).
__device__ __forceinline__ uint4 lds_u128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
  return v;
}
__device__ __forceinline__ float4 lds_f128(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(addr));
  return v;
}
__device__ __forceinline__ uint32_t lds_u32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr));
  return v;
}

// Packed bf16 arithmetic on two lanes (low half, high half), one rounding each.
__device__ __forceinline__ uint32_t bf16x2_mul(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ uint32_t bf16x2_fma(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("fma.rn.bf16x2 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}
__device__ __forceinline__ uint32_t bf16x2_neg(uint32_t a) {
  uint32_t d;
  asm("neg.bf16x2 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}
// x * v as hi + lo (bf16 pairs) for a weight given as whi + wlo (bf16 pairs):
// hi = RN(whi v); the residual whi v - hi has at most 8 significant bits and is
// exact in bf16 (one fused multiply-add); lo = RN(wlo v + residual).
// |hi + lo - (whi + wlo) v| <= 2^-9 |lo| ~ 2^-17 |x v|.
__device__ __forceinline__ void bf16x2_scale_split(uint32_t whi, uint32_t wlo, uint32_t v, uint32_t& hi,
                                                   uint32_t& lo) {
  hi = bf16x2_mul(whi, v);
  lo = bf16x2_fma(wlo, v, bf16x2_fma(whi, v, bf16x2_neg(hi)));
}

}  // namespace jacap
