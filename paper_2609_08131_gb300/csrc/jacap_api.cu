// jacap_api.cu - host side of the libjacap C ABI (declared in include/jacap.h).
//
// Validates arguments on the host before anything is enqueued, carves the
// caller's workspace, encodes the TMA tensor maps of K and V, and enqueues the
// kernels of the eviction pass on the caller's stream. Allocates nothing.
#include <algorithm>
#include <cudaTypedefs.h>
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "jacap.h"
#include "jacap_dev.cuh"
#include "jacap_internal.h"

using namespace jacap;

namespace {

constexpr size_t ALIGN = 1024;
inline size_t align_up(size_t x) { return (x + ALIGN - 1) & ~(ALIGN - 1); }

struct Carve {
  size_t status, plan, chunks, counters, mu, lam, qdev, lk, cstats, ustats, w, gpart, pflag, gram, minv,
      minv_img, total;
  size_t units, trace, trace_cta;
};

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// Argument checks that need no GPU. Returns JACAP_OK or the error.
jacap_status check_layout(const jacap_layout* L) {
  if (L == nullptr || L->cu_seqlens == nullptr) return JACAP_ERR_INVALID_ARG;
  if (L->num_seqs < 1 || L->num_layers < 1 || L->num_kv_heads < 1 || L->num_q_heads < 1) return JACAP_ERR_INVALID_ARG;
  if (L->total_tokens < 1 || L->total_tokens >= ((int64_t)1 << 31)) return JACAP_ERR_INVALID_ARG;
  if (L->max_seqlen < 1 || (int64_t)L->max_seqlen > L->total_tokens) return JACAP_ERR_INVALID_ARG;
  if (L->window < 1) return JACAP_ERR_INVALID_ARG;
  if (L->dtype != JACAP_F32 && L->dtype != JACAP_BF16) return JACAP_ERR_INVALID_ARG;
  if (L->num_q_heads % L->num_kv_heads != 0) return JACAP_ERR_INVALID_ARG;
  const int G = L->num_q_heads / L->num_kv_heads;
  if (L->head_dim != D) return JACAP_ERR_UNSUPPORTED;
  if (G > G_MAX) return JACAP_ERR_UNSUPPORTED;
  const int64_t el16 = L->dtype == JACAP_BF16 ? 8 : 4;  // elements per 16 bytes
  const int64_t kv[3] = {L->kv_stride_layer, L->kv_stride_head, L->kv_stride_token};
  const int64_t qs[4] = {L->q_stride_seq, L->q_stride_layer, L->q_stride_head, L->q_stride_pos};
  for (int64_t s : kv)
    if (s < D || s % el16 != 0) return JACAP_ERR_INVALID_ARG;
  for (int64_t s : qs)
    if (s < D || s % el16 != 0) return JACAP_ERR_INVALID_ARG;
  const int64_t es = L->dtype == JACAP_BF16 ? 2 : 4;
  if ((uint64_t)L->kv_stride_layer * es >= (1ull << 40) || (uint64_t)L->kv_stride_head * es >= (1ull << 40) ||
      (uint64_t)L->kv_stride_token * es >= (1ull << 40))
    return JACAP_ERR_INVALID_ARG;
  return JACAP_OK;
}

// Tokens per work item: the largest of 16384..128 that still yields 4096
// items (independent of the device so the workspace size is a pure function
// of the layout). Each CTA takes a contiguous range of items, so the counts
// per CTA differ by one item at most: with ~27 items per CTA on 152 SMs the
// last item costs under 4 % of a pass. Items of one unit that follow each
// other in a CTA's range share one partial Gram and one factor image.
#ifndef JACAP_TARGET_ITEMS
#define JACAP_TARGET_ITEMS 4096
#endif
int pick_chunk(const jacap_layout* L) {
  const int64_t planes = (int64_t)L->num_layers * L->num_kv_heads;
  for (int c = 16384; c > TILE; c >>= 1) {
    const int64_t items = planes * (L->total_tokens / c + L->num_seqs);
    if (items >= JACAP_TARGET_ITEMS) return c;
  }
  return TILE;
}

void make_dims(const jacap_layout* L, const jacap_params* P, Dims& dm) {
  memset(&dm, 0, sizeof(dm));
  dm.pdl = 1;
  dm.S = L->num_seqs;
  dm.L = L->num_layers;
  dm.Hq = L->num_q_heads;
  dm.Hkv = L->num_kv_heads;
  dm.G = L->num_q_heads / L->num_kv_heads;
  dm.window = L->window;
  dm.Ntot = L->total_tokens;
  dm.chunk = pick_chunk(L);
  dm.c_cap = L->total_tokens / dm.chunk + L->num_seqs;
  dm.kv_sl = L->kv_stride_layer;
  dm.kv_sh = L->kv_stride_head;
  dm.kv_st = L->kv_stride_token;
  dm.q_ss = L->q_stride_seq;
  dm.q_sl = L->q_stride_layer;
  dm.q_sh = L->q_stride_head;
  dm.q_sp = L->q_stride_pos;
  if (P != nullptr) {
    dm.inv_scale = (float)(1.0 / ((double)P->tau * sqrt((double)D)));
    dm.wdiv = P->weight_div_dk ? 1.0f / (float)D : 1.0f;
    dm.cov_unbiased = P->cov_unbiased;
    dm.linear = P->linear_weighting;
    dm.full_cov = P->full_covariance;
    if (dm.full_cov && L->dtype == JACAP_BF16) dm.kf_rp = kfull_rows_padded(dm.G, dm.window);
  }
}

Carve carve(const Dims& dm) {
  Carve c;
  const size_t planes = (size_t)dm.L * dm.Hkv;
  const size_t units = planes * dm.S;
  size_t o = 0;
  c.units = units;
  c.status = o; o = align_up(o + 64);
  c.plan = o; o = align_up(o + ((size_t)dm.S + 2) * 4);
  c.chunks = o; o = align_up(o + (size_t)dm.c_cap * 16);
  c.counters = o; o = align_up(o + units * 8);  // gcount and fdone of the fused schedule
  c.mu = o; o = align_up(o + (size_t)dm.S * dm.L * dm.Hq * D * 4);
  c.lam = o; o = align_up(o + (size_t)dm.S * dm.L * dm.Hq * D * 4);
  // centred window queries: fp32 rows, or the bf16 hi/lo image (512 bytes per padded row)
  const size_t qrows = std::max((size_t)dm.G * dm.window, (size_t)kfull_rows_padded(dm.G, dm.window));
  c.qdev = o; o = align_up(o + (size_t)dm.S * dm.L * dm.Hkv * qrows * 512);
  c.lk = o; o = align_up(o + planes * (size_t)dm.Ntot * 2 * dm.G * 4 + 16);  // + tail of 16-byte rounded copies
  c.cstats = o; o = align_up(o + planes * (size_t)dm.c_cap * dm.G * 2 * 4);
  c.ustats = o; o = align_up(o + units * (size_t)dm.G * 2 * 4);
  c.w = o; o = align_up(o + planes * (size_t)dm.Ntot * 4);
  c.gpart = o; o = align_up(o + planes * (size_t)dm.c_cap * D * D * 4);
  c.pflag = o; o = align_up(o + planes * (size_t)dm.c_cap * 4);
  c.gram = o; o = align_up(o + units * D * D * 4);
  c.minv = o; o = align_up(o + units * D * D * 4);
  c.minv_img = o; o = align_up(o + units * 65536);
#ifdef JACAP_TRACE
  c.trace = o; o = align_up(o + units * TR_SLOTS * 8);  // trace builds: the fused schedule's timeline,
  c.trace_cta = o; o = align_up(o + (size_t)TR_KERNELS * TR_CTAS * TR_CTA_SLOTS * 8);  // then the CTA accounting
#else
  c.trace = 0;
  c.trace_cta = 0;
#endif
  c.total = o;
  return c;
}

Ws make_ws(void* base, const Carve& c) {
  uint8_t* b = (uint8_t*)base;
  Ws ws;
  ws.status = (uint32_t*)(b + c.status);
  ws.plan = (int32_t*)(b + c.plan);
  ws.chunks = (int4*)(b + c.chunks);
  ws.gcount = (int32_t*)(b + c.counters);
  ws.fdone = ws.gcount + c.units;  // right after gcount: the plan kernel zeroes 2 x units words
  ws.mu = (float*)(b + c.mu);
  ws.lam = (float*)(b + c.lam);
  ws.qdev = (float*)(b + c.qdev);
  ws.qimg = b + c.qdev;
  ws.lk = (float*)(b + c.lk);
  ws.cstats = (float*)(b + c.cstats);
  ws.ustats = (float*)(b + c.ustats);
  ws.w = (float*)(b + c.w);
  ws.gpart = (float*)(b + c.gpart);
  ws.pflag = (int32_t*)(b + c.pflag);
  ws.gram = (float*)(b + c.gram);
  ws.minv = (float*)(b + c.minv);
  ws.minv_img = b + c.minv_img;
  ws.trace = c.trace != 0 ? (unsigned long long*)(b + c.trace) : nullptr;
  ws.trace_cta = c.trace_cta != 0 ? (unsigned long long*)(b + c.trace_cta) : nullptr;
  return ws;
}

// Current device must be sm_103 (GB300). Returns its SM count via *sms.
jacap_status check_device(int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return JACAP_ERR_CUDA;
  int major = 0, minor = 0;
  if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return JACAP_ERR_CUDA;
  if (major != 10 || minor != 3) return JACAP_ERR_UNSUPPORTED;
  return JACAP_OK;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = (PFN_cuTensorMapEncodeTiled_v12000)p;
  }
  return fn;
}

// 4-D map over (channel, token, kv head, layer) with {128 B, 128 tokens} boxes
// and the 128-byte swizzle; out-of-range tokens read as zero.
bool encode_kv_map(CUtensorMap* map, const jacap_layout* L, const void* base) {
  PFN_cuTensorMapEncodeTiled_v12000 fn = encode_fn();
  if (fn == nullptr) return false;
  const bool bf = L->dtype == JACAP_BF16;
  const cuuint64_t es = bf ? 2 : 4;
  const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)L->total_tokens, (cuuint64_t)L->num_kv_heads,
                              (cuuint64_t)L->num_layers};
  const cuuint64_t strides[3] = {(cuuint64_t)L->kv_stride_token * es, (cuuint64_t)L->kv_stride_head * es,
                                 (cuuint64_t)L->kv_stride_layer * es};
  const cuuint32_t box[4] = {(cuuint32_t)(128 / es), (cuuint32_t)TILE, 1, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  const CUresult r = fn(map, bf ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4,
                        const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

jacap_status map_cuda(cudaError_t e) { return e == cudaSuccess ? JACAP_OK : JACAP_ERR_CUDA; }

// The per-token tags `pos` follow K's layer and head strides in units of its
// token stride, which must therefore divide them.
bool pos_layout_ok(const jacap_layout* L, const int32_t* pos) {
  return pos == nullptr || (L->kv_stride_layer % L->kv_stride_token == 0 && L->kv_stride_head % L->kv_stride_token == 0);
}

// CTAs for `items` work items with at most per_sm CTAs per SM: each CTA takes
// a contiguous range, so the grid is chosen to split the items as evenly as
// the cap allows (ceil(items / cap) items for every CTA but the last few).
int persistent_grid(int64_t items, int sms, int per_sm) {
  const int64_t cap = (int64_t)sms * per_sm;
  if (items <= cap) return items < 1 ? 1 : (int)items;
  const int64_t per = (items + cap - 1) / cap;
  return (int)((items + per - 1) / per);
}

// The fused schedule (k_fused.cu). Cost model in SM-microseconds: a 128-token
// tile costs the Gram role its 16 MMAs of N = 128 (1024 tensor cycles) and
// the score role its MMAs (SC_TILE_CYCLES), both at ~1.7 G useful cycles/s;
// a factor CTA takes ~30 us per unit. The factor role gets enough CTAs to
// keep pace (at most a quarter of the SMs), the rest split between Gram and
// score in proportion to their cost per tile.
constexpr double FU_GRAM_US = 1024.0 / 1700.0;
constexpr double FU_SCORE_US = 880.0 / 1700.0;
constexpr double FU_FACTOR_US = 30.0;

double fused_tiles(const jacap_layout* L, const Dims& dm) {
  return (double)dm.L * dm.Hkv * ((double)L->total_tokens / TILE + 0.5 * dm.S);
}

FusedRoles fused_roles(const jacap_layout* L, const Dims& dm, int sms) {
  const double units = (double)dm.L * dm.Hkv * dm.S, tiles = fused_tiles(L, dm);
  int nf = 1;
  for (int iter = 0; iter < 4; ++iter) {
    const double t = tiles * (FU_GRAM_US + FU_SCORE_US) / (sms - nf);
    nf = std::min(std::max((int)ceil(units * FU_FACTOR_US / t), 1), sms / 4);
  }
  const int rest = sms - nf;
  const int ng = std::min(std::max((int)lround(rest * FU_GRAM_US / (FU_GRAM_US + FU_SCORE_US)), 1), rest - 1);
  FusedRoles r{nf, ng, rest - ng};
  // tuning override: JACAP_FUSED_ROLES="nf,ng" (the score role takes the other SMs)
  if (const char* e = getenv("JACAP_FUSED_ROLES")) {
    int a = 0, b = 0;
    if (sscanf(e, "%d,%d", &a, &b) == 2 && a >= 1 && b >= 1 && a + b < sms) r = FusedRoles{a, b, sms - a - b};
  }
  return r;
}

// V tiles per Gram item left in L2 (evict_last) for the score role: the
// evict_last lines in flight (about ng + ns items and nf units' worth of
// items) stay within 60 % of L2.
int fused_keep_tiles(const Dims& dm, const FusedRoles& r, double items_per_unit) {
  int dev = 0, l2 = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev) != cudaSuccess)
    l2 = 0;
  const double span = r.ng + r.ns + r.nf * items_per_unit;  // items whose kept tiles are in flight
  int keep = (int)(0.6 * l2 / (span * 32768.0));
  if (const char* e = getenv("JACAP_KEEP_TILES")) keep = atoi(e);  // tuning override (< 0: no L2 hints)
  return std::min(std::max(keep, -1), dm.chunk / TILE);
}

// Items a fused-role CTA takes at a time: about 8 partial Grams per unit for
// the factor to sum, runs of at most 8192 tokens (a unit's items should finish
// close in time, for L2).
int fused_run_items(const Dims& dm, double items_per_unit) {
  const int by_parts = (int)(items_per_unit / 8.0);
  int r = std::max(1, std::min(by_parts, 8192 / dm.chunk));
  if (const char* e = getenv("JACAP_RUN_ITEMS")) r = std::max(1, atoi(e));  // tuning override
  return r;
}

// The automatic choice is the separate kernels. Measured on GB300 (config 2:
// 32 layers x 8 KV heads, n = 32768) the fused launch takes 0.96 ms against
// 0.80 ms for the Gram, the factor and the scores apart: a unit stays ~150 us
// between its first Gram tile and its last score tile, so at the pass's rate
// of V far more than L2 is in flight and only ~12 % of the second read hits
// L2, while the roles' fill and drain (~80 us each) add to a pass whose
// separate kernels already run at the effective HBM rate.
bool fused_pays(const jacap_layout*, const Dims&, int) { return false; }

// 2 (fused, with its roles and kept tiles) or 1 (separate kernels) for a
// validated layout and params.
int pick_schedule(const jacap_layout* L, const jacap_params* P, const Dims& dm, int sms, bool dense,
                  FusedRoles* roles, int* keep, int* run) {
  const bool fused = L->dtype == JACAP_BF16 && !dense && sms >= 8 &&
                     (P->schedule == 2 || (P->schedule == 0 && fused_pays(L, dm, sms)));
  if (!fused) return 1;
  *roles = fused_roles(L, dm, sms);
  const double per_plane =
      L->num_seqs == 1 ? ceil((double)L->total_tokens / dm.chunk) : (double)L->total_tokens / dm.chunk + 0.5 * dm.S;
  *keep = fused_keep_tiles(dm, *roles, per_plane / dm.S);
  *run = fused_run_items(dm, per_plane / dm.S);
  return 2;
}

// Work items of the pass (plane x chunk): exact for one request, otherwise the
// capacity bound (the device computes the exact count from cu_seqlens).
int64_t pass_items(const jacap_layout* L, const Dims& dm) {
  const int64_t per_plane = L->num_seqs == 1 ? (L->total_tokens + dm.chunk - 1) / dm.chunk : dm.c_cap;
  return (int64_t)dm.L * dm.Hkv * per_plane;
}

}  // namespace

extern "C" {

size_t jacap_workspace_size(const jacap_layout* layout, int32_t budget) {
  if (check_layout(layout) != JACAP_OK || budget < 1) return 0;
  Dims dm;
  make_dims(layout, nullptr, dm);
  return carve(dm).total;
}

jacap_status jacap_workspace_offsets(const jacap_layout* layout, int32_t budget, jacap_ws_offsets* out) {
  if (out == nullptr || budget < 1) return JACAP_ERR_INVALID_ARG;
  const jacap_status st = check_layout(layout);
  if (st != JACAP_OK) return st;
  Dims dm;
  make_dims(layout, nullptr, dm);
  const Carve c = carve(dm);
  out->mu_scaled = c.mu;
  out->lambda = c.lam;
  out->weights = c.w;
  out->gram = c.gram;
  out->chol_inv = c.minv;
  out->trace_timeline = c.trace;
  out->trace_cta = c.trace_cta;
  return JACAP_OK;
}

jacap_status jacap_score(const jacap_layout* layout, const jacap_params* params, const void* q_win,
                         const void* k, const void* v, float* scores, void* ws, size_t ws_bytes, void* stream) {
  return jacap_score_timed(layout, params, q_win, k, v, scores, ws, ws_bytes, stream, nullptr, 0);
}

jacap_status jacap_score_timed(const jacap_layout* layout, const jacap_params* params, const void* q_win,
                               const void* k, const void* v, float* scores, void* ws, size_t ws_bytes,
                               void* stream, void* const* events, int32_t num_events) {
  return jacap_score_out(layout, params, q_win, k, v, nullptr, scores, ws, ws_bytes, stream, events, num_events);
}

}  // extern "C"

namespace {

// The scoring pass behind jacap_score_out (query statistics from q_win) and
// jacap_score_stats (from running statistics: stats != NULL, q_win unused).
jacap_status score_pass(const jacap_layout* layout, const jacap_params* params, const void* q_win,
                        const float* stats, const int32_t* counts, const void* k, const void* v,
                        const float* out_factor, float* scores, void* ws, size_t ws_bytes, void* stream,
                        void* const* events, int32_t num_events) {
  if (num_events != 0 && (num_events != JACAP_SCORE_KERNELS + 1 || events == nullptr)) return JACAP_ERR_INVALID_ARG;
  jacap_status st = check_layout(layout);
  if (st != JACAP_OK) return st;
  const bool running = stats != nullptr;
  if (params == nullptr || (!running && q_win == nullptr) || (running && counts == nullptr) || k == nullptr ||
      v == nullptr || scores == nullptr || ws == nullptr)
    return JACAP_ERR_INVALID_ARG;
  if (!(params->tau > 0.f) || !isfinite(params->tau)) return JACAP_ERR_INVALID_ARG;
  if (params->weight_div_dk != 0 && params->weight_div_dk != 1) return JACAP_ERR_INVALID_ARG;
  if (params->cov_unbiased != 0 && params->cov_unbiased != 1) return JACAP_ERR_INVALID_ARG;
  if (!running && params->cov_unbiased && layout->window < 2) return JACAP_ERR_INVALID_ARG;
  if (params->linear_weighting != 0 && params->linear_weighting != 1) return JACAP_ERR_INVALID_ARG;
  if (params->full_covariance != 0 && params->full_covariance != 1) return JACAP_ERR_INVALID_ARG;
  if (params->schedule < 0 || params->schedule > 2) return JACAP_ERR_INVALID_ARG;
  if (params->ridge != 1 || (running && params->full_covariance != 0)) return JACAP_ERR_UNSUPPORTED;
  if ((!running && !aligned16(q_win)) || !aligned16(k) || !aligned16(v) || ((uintptr_t)scores & 3u) != 0 ||
      (out_factor != nullptr && !aligned16(out_factor)) || (running && (!aligned16(stats) || ((uintptr_t)counts & 3u))))
    return JACAP_ERR_INVALID_ARG;
  Dims dm;
  make_dims(layout, params, dm);
  dm.dense_minv = out_factor != nullptr ? 1 : 0;
  dm.pdl = num_events == 0 ? 1 : 0;  // timing events between kernels serialise them anyway
  const Carve c = carve(dm);
  if (((uintptr_t)ws & 255u) != 0 || ws_bytes < c.total) return JACAP_ERR_WORKSPACE;
  int sms = 0;
  if ((st = check_device(&sms)) != JACAP_OK) return st;
  cudaStream_t s = (cudaStream_t)stream;
  const Ws w = make_ws(ws, c);
  CUtensorMap kmap, vmap;
  const bool bf = layout->dtype == JACAP_BF16;
  if (!encode_kv_map(&kmap, layout, k) || !encode_kv_map(&vmap, layout, v)) return JACAP_ERR_CUDA;
  const int64_t items = pass_items(layout, dm);
  const int dt = bf ? 1 : 0;
  const int32_t* cu = layout->cu_seqlens;
  // hook(i): the boundary before kernel i (optional timing event; with
  // -DJACAP_NVTX the end of kernel i-1's trace range and the start of i's)
  static const char* const kTrace[JACAP_SCORE_KERNELS] = {"jacap/plan",  "jacap/query_stats", "jacap/k_pass",
                                                          "jacap/weights", "jacap/gram",      "jacap/factor",
                                                          "jacap/scores"};
  int traced = -1;
  auto hook = [&](int i) -> jacap_status {
    if (traced >= 0) trace_pop();
    traced = -1;
    if (i < JACAP_SCORE_KERNELS) {
      trace_push(kTrace[i]);
      traced = i;
    }
    if (num_events == 0) return JACAP_OK;
    return map_cuda(cudaEventRecord((cudaEvent_t)events[i], s));
  };
  struct TraceGuard {  // closes an open range on an early return
    int& t;
    ~TraceGuard() {
      if (t >= 0) trace_pop();
    }
  } trace_guard{traced};
  if ((st = hook(0)) != JACAP_OK || (st = map_cuda(launch_plan(dm, w, cu, s))) != JACAP_OK) return st;
  if ((st = hook(1)) != JACAP_OK ||
      (st = map_cuda(running ? launch_stats_moments(dm, w, stats, counts, s)
                             : launch_window_stats(dm, w, dt, q_win, s))) != JACAP_OK)
    return st;
  // full covariance on the tensor cores: one kernel does the K pass with that kappa
  const bool fused_full = dm.full_cov && kfull_uses_tensor_cores(dm, dt);
  if ((st = hook(2)) != JACAP_OK ||
      (st = map_cuda(fused_full ? launch_kpass_full(kmap, dm, w, persistent_grid(items, sms, 1), s)
                                : launch_kpass(kmap, dm, w, dt, cu, persistent_grid(items, sms, 1), s))) != JACAP_OK)
    return st;
  if (dm.full_cov && !fused_full &&  // overwrites the K pass's diagonal kappa; timed with the K pass
      (st = map_cuda(launch_kfull(kmap, dm, w, dt, k, persistent_grid(items, sms, 2), s))) != JACAP_OK)
    return st;
  // each unit's softmax normaliser from the K pass's chunk statistics (timed with the weights)
  if ((st = hook(3)) != JACAP_OK || (st = map_cuda(launch_unit_stats(dm, w, s))) != JACAP_OK) return st;
  FusedRoles roles{0, 0, 0};
  int keep = 0, run = 1;
  if (pick_schedule(layout, params, dm, sms, out_factor != nullptr, &roles, &keep, &run) == 2) {
    // the Gram, the factor and the scores in one launch (timed as the Gram)
    Dims fd = dm;
    fd.fused = 1;
    fd.keep_tiles = keep;
    fd.run_items = run;
    if ((st = hook(4)) != JACAP_OK ||
        (st = map_cuda(launch_fused(vmap, fd, w, scores, roles, s))) != JACAP_OK || (st = hook(5)) != JACAP_OK ||
        (st = hook(6)) != JACAP_OK || (st = hook(7)) != JACAP_OK)
      return st;
    return JACAP_OK;
  }
  // (bf16 caches: the Gram kernel computes the weights from the K pass's rows)
  if (!bf && (st = map_cuda(launch_weights(dm, w, cu, persistent_grid(items, sms, 8), s))) != JACAP_OK) return st;
  if ((st = hook(4)) != JACAP_OK ||
      (st = map_cuda(launch_gram(vmap, dm, w, dt, v, cu, persistent_grid(items, sms, bf ? 1 : 4), s))) != JACAP_OK)
    return st;
  if ((st = hook(5)) != JACAP_OK || (st = map_cuda(launch_factor(dm, w, out_factor, s))) != JACAP_OK) return st;
  if ((st = hook(6)) != JACAP_OK ||
      (st = map_cuda(launch_score(vmap, dm, w, dt, v, cu, scores, persistent_grid(items, sms, bf ? 1 : 2), s))) !=
          JACAP_OK)
    return st;
  if ((st = hook(7)) != JACAP_OK) return st;
  return JACAP_OK;
}

}  // namespace

extern "C" {

jacap_status jacap_score_out(const jacap_layout* layout, const jacap_params* params, const void* q_win,
                             const void* k, const void* v, const float* out_factor, float* scores, void* ws,
                             size_t ws_bytes, void* stream, void* const* events, int32_t num_events) {
  return score_pass(layout, params, q_win, nullptr, nullptr, k, v, out_factor, scores, ws, ws_bytes, stream, events,
                    num_events);
}

int32_t jacap_schedule_info(const jacap_layout* layout, const jacap_params* params, int32_t* roles) {
  jacap_status st = check_layout(layout);
  if (st != JACAP_OK) return -(int32_t)st;
  if (params == nullptr || params->schedule < 0 || params->schedule > 2) return -(int32_t)JACAP_ERR_INVALID_ARG;
  int sms = 0;
  if ((st = check_device(&sms)) != JACAP_OK) return -(int32_t)st;
  Dims dm;
  make_dims(layout, params, dm);
  FusedRoles r{0, 0, 0};
  int keep = 0, run = 1;
  const int sched = pick_schedule(layout, params, dm, sms, false, &r, &keep, &run);
  if (roles != nullptr) {
    roles[0] = r.nf;
    roles[1] = r.ng;
    roles[2] = r.ns;
    roles[3] = keep;
  }
  return sched;
}

jacap_status jacap_score_stats(const jacap_layout* layout, const jacap_params* params, const float* stats,
                               const int32_t* counts, const void* k, const void* v, float* scores, void* ws,
                               size_t ws_bytes, void* stream, void* const* events, int32_t num_events) {
  if (stats == nullptr) return JACAP_ERR_INVALID_ARG;
  return score_pass(layout, params, nullptr, stats, counts, k, v, nullptr, scores, ws, ws_bytes, stream, events,
                    num_events);
}

jacap_status jacap_stats_update(const jacap_layout* layout, const void* q_new, int32_t reset, float* stats,
                                int32_t* counts, void* stream) {
  jacap_status st = check_layout(layout);
  if (st != JACAP_OK) return st;
  if (q_new == nullptr || stats == nullptr || counts == nullptr || (reset != 0 && reset != 1))
    return JACAP_ERR_INVALID_ARG;
  if (!aligned16(q_new) || !aligned16(stats) || ((uintptr_t)counts & 3u) != 0) return JACAP_ERR_INVALID_ARG;
  int sms = 0;
  if ((st = check_device(&sms)) != JACAP_OK) return st;
  Dims dm;
  make_dims(layout, nullptr, dm);
  return map_cuda(launch_stats_update(dm, layout->dtype == JACAP_BF16 ? 1 : 0, q_new, stats, counts, reset,
                                      (cudaStream_t)stream));
}

jacap_status jacap_compact_inplace(const jacap_layout* layout, void* k, void* v, int32_t* pos, const int32_t* idx,
                                   int32_t budget, int32_t preserve_order, void* ws, size_t ws_bytes, void* stream) {
  jacap_status st = check_layout(layout);
  if (st != JACAP_OK) return st;
  if (k == nullptr || v == nullptr || idx == nullptr || ws == nullptr || budget < 1 ||
      (preserve_order != 0 && preserve_order != 1))
    return JACAP_ERR_INVALID_ARG;
  if (!aligned16(k) || !aligned16(v) || ((uintptr_t)idx & 3u) != 0 || ((uintptr_t)pos & 3u) != 0)
    return JACAP_ERR_INVALID_ARG;
  if (!pos_layout_ok(layout, pos)) return JACAP_ERR_INVALID_ARG;
  if ((int64_t)layout->num_layers * layout->num_kv_heads * layout->num_seqs >= ((int64_t)1 << 31))
    return JACAP_ERR_INVALID_ARG;
  Dims dm;
  make_dims(layout, nullptr, dm);
  const Carve c = carve(dm);
  if (((uintptr_t)ws & 255u) != 0 || ws_bytes < c.total) return JACAP_ERR_WORKSPACE;
  int sms = 0;
  if ((st = check_device(&sms)) != JACAP_OK) return st;
  return map_cuda(launch_compact_inplace(dm, make_ws(ws, c), layout->dtype == JACAP_BF16 ? 1 : 0,
                                         layout->cu_seqlens, k, v, pos, idx, budget, preserve_order,
                                         (cudaStream_t)stream));
}

jacap_status jacap_select_compact_inplace(const jacap_layout* layout, const float* scores, int32_t budget,
                                          int32_t* idx, int32_t* kept, void* k, void* v, int32_t* pos,
                                          int32_t preserve_order, void* ws, size_t ws_bytes, void* stream) {
  jacap_status st = check_layout(layout);
  if (st != JACAP_OK) return st;
  if (scores == nullptr || idx == nullptr || kept == nullptr || k == nullptr || v == nullptr || ws == nullptr ||
      budget < 1 || (preserve_order != 0 && preserve_order != 1))
    return JACAP_ERR_INVALID_ARG;
  if (((uintptr_t)scores & 3u) != 0 || ((uintptr_t)idx & 3u) != 0 || ((uintptr_t)kept & 3u) != 0 ||
      ((uintptr_t)pos & 3u) != 0 || !aligned16(k) || !aligned16(v))
    return JACAP_ERR_INVALID_ARG;
  if (!pos_layout_ok(layout, pos)) return JACAP_ERR_INVALID_ARG;
  Dims dm;
  make_dims(layout, nullptr, dm);
  const Carve c = carve(dm);
  if (((uintptr_t)ws & 255u) != 0 || ws_bytes < c.total) return JACAP_ERR_WORKSPACE;
  int sms = 0;
  if ((st = check_device(&sms)) != JACAP_OK) return st;
  const Ws w = make_ws(ws, c);
  const int64_t units = (int64_t)dm.L * dm.Hkv * dm.S;
  const int dt = layout->dtype == JACAP_BF16 ? 1 : 0;
  const cudaStream_t s = (cudaStream_t)stream;
  const TraceRange trace("jacap/select_compact_inplace");
  if (!preserve_order)  // hole filling inside the selection kernel
    return map_cuda(launch_select(dm, w, layout->cu_seqlens, scores, budget, idx, kept, layout->max_seqlen,
                                  persistent_grid(units, sms, 2), s, dt, nullptr, nullptr, nullptr, nullptr, k, v,
                                  pos));
  // ascending order moves every kept row: its own launch after the selection
  if ((st = map_cuda(launch_select(dm, w, layout->cu_seqlens, scores, budget, idx, kept, layout->max_seqlen,
                                   persistent_grid(units, sms, 2), s))) != JACAP_OK)
    return st;
  return map_cuda(launch_compact_inplace(dm, w, dt, layout->cu_seqlens, k, v, pos, idx, budget, 1, s));
}

jacap_status jacap_select(const jacap_layout* layout, const float* scores, int32_t budget, int32_t* idx,
                          int32_t* kept, void* ws, size_t ws_bytes, void* stream) {
  jacap_status st = check_layout(layout);
  if (st != JACAP_OK) return st;
  if (scores == nullptr || idx == nullptr || kept == nullptr || ws == nullptr || budget < 1)
    return JACAP_ERR_INVALID_ARG;
  if (((uintptr_t)scores & 3u) != 0 || ((uintptr_t)idx & 3u) != 0 || ((uintptr_t)kept & 3u) != 0)
    return JACAP_ERR_INVALID_ARG;
  Dims dm;
  make_dims(layout, nullptr, dm);
  const Carve c = carve(dm);
  if (((uintptr_t)ws & 255u) != 0 || ws_bytes < c.total) return JACAP_ERR_WORKSPACE;
  int sms = 0;
  if ((st = check_device(&sms)) != JACAP_OK) return st;
  const Ws w = make_ws(ws, c);
  const int64_t units = (int64_t)dm.L * dm.Hkv * dm.S;
  const TraceRange trace("jacap/select");
  return map_cuda(launch_select(dm, w, layout->cu_seqlens, scores, budget, idx, kept, layout->max_seqlen,
                                persistent_grid(units, sms, 2), (cudaStream_t)stream));
}

jacap_status jacap_select_compact(const jacap_layout* layout, const float* scores, int32_t budget, int32_t* idx,
                                  int32_t* kept, const void* k, const void* v, void* k_out, void* v_out, void* ws,
                                  size_t ws_bytes, void* stream) {
  jacap_status st = check_layout(layout);
  if (st != JACAP_OK) return st;
  if (scores == nullptr || idx == nullptr || kept == nullptr || ws == nullptr || budget < 1 || k == nullptr ||
      v == nullptr || k_out == nullptr || v_out == nullptr)
    return JACAP_ERR_INVALID_ARG;
  if (((uintptr_t)scores & 3u) != 0 || ((uintptr_t)idx & 3u) != 0 || ((uintptr_t)kept & 3u) != 0)
    return JACAP_ERR_INVALID_ARG;
  if (!aligned16(k) || !aligned16(v) || !aligned16(k_out) || !aligned16(v_out)) return JACAP_ERR_INVALID_ARG;
  Dims dm;
  make_dims(layout, nullptr, dm);
  const Carve c = carve(dm);
  if (((uintptr_t)ws & 255u) != 0 || ws_bytes < c.total) return JACAP_ERR_WORKSPACE;
  int sms = 0;
  if ((st = check_device(&sms)) != JACAP_OK) return st;
  const Ws w = make_ws(ws, c);
  const int64_t units = (int64_t)dm.L * dm.Hkv * dm.S;
  const TraceRange trace("jacap/select_compact");
  return map_cuda(launch_select(dm, w, layout->cu_seqlens, scores, budget, idx, kept, layout->max_seqlen,
                                persistent_grid(units, sms, 2), (cudaStream_t)stream,
                                layout->dtype == JACAP_BF16 ? 1 : 0, k, v, k_out, v_out));
}

jacap_status jacap_compact(const jacap_layout* layout, const void* k, const void* v, const int32_t* idx,
                           int32_t budget, void* k_out, void* v_out, void* stream) {
  jacap_status st = check_layout(layout);
  if (st != JACAP_OK) return st;
  if (k == nullptr || v == nullptr || idx == nullptr || k_out == nullptr || v_out == nullptr || budget < 1)
    return JACAP_ERR_INVALID_ARG;
  if (!aligned16(k) || !aligned16(v) || !aligned16(k_out) || !aligned16(v_out) || ((uintptr_t)idx & 3u) != 0)
    return JACAP_ERR_INVALID_ARG;
  int sms = 0;
  if ((st = check_device(&sms)) != JACAP_OK) return st;
  Dims dm;
  make_dims(layout, nullptr, dm);
  const TraceRange trace("jacap/compact");
  return map_cuda(launch_compact(dm, layout->dtype == JACAP_BF16 ? 1 : 0, layout->cu_seqlens, k, v, idx, budget,
                                 k_out, v_out, (cudaStream_t)stream));
}

jacap_status jacap_selftest_wait(void* ws, size_t ws_bytes, int64_t limit_ns, void* stream) {
  if (ws == nullptr || ((uintptr_t)ws & 255u) != 0 || ws_bytes < 64) return JACAP_ERR_INVALID_ARG;
  if (limit_ns < 1000 || limit_ns > 10000000000LL) return JACAP_ERR_INVALID_ARG;
  int sms = 0;
  jacap_status st = check_device(&sms);
  if (st != JACAP_OK) return st;
  Ws w;
  memset(&w, 0, sizeof(w));
  w.status = (uint32_t*)ws;
  return map_cuda(launch_selftest_wait(w, (unsigned long long)limit_ns, (cudaStream_t)stream));
}

jacap_status jacap_device_status(const void* ws, void* stream) {
  if (ws == nullptr) return JACAP_ERR_INVALID_ARG;
  if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return JACAP_ERR_CUDA;
  uint32_t word = 0;
  if (cudaMemcpy(&word, ws, sizeof(word), cudaMemcpyDeviceToHost) != cudaSuccess) return JACAP_ERR_CUDA;
  if (word & ST_INVALID) return JACAP_ERR_INVALID_ARG;
  if (word & ST_TIMEOUT) return JACAP_ERR_TIMEOUT;
  if (word & ST_NONFINITE) return JACAP_ERR_NONFINITE;
  return JACAP_OK;
}

const char* jacap_status_string(jacap_status status) {
  switch (status) {
    case JACAP_OK: return "ok";
    case JACAP_ERR_INVALID_ARG: return "invalid argument";
    case JACAP_ERR_UNSUPPORTED: return "unsupported configuration or device";
    case JACAP_ERR_WORKSPACE: return "workspace too small or misaligned";
    case JACAP_ERR_CUDA: return "CUDA runtime or launch error";
    case JACAP_ERR_NONFINITE: return "non-finite value in an input or intermediate";
    case JACAP_ERR_TIMEOUT: return "a bounded device wait expired";
    default: return "unknown status";
  }
}

}  // extern "C"
