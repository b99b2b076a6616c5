// jacap_host.cu - eviction of a KV cache held in host memory (declared in
// include/jacap.h): jacap_host_buffer_size and jacap_evict_host.
//
// An offloaded cache (the KV cache of Sec. 3.1 kept in host memory) reaches
// the device in groups of layers through two device buffers inside the
// caller's device buffer: while the pass (Algorithm 1 steps 1-5 and the
// compaction into the retained cache Z_C) runs over group g on `stream`, group
// g + 1 is copied host -> device on `copy_stream`, so the device never holds
// more than two groups and the pass overlaps the copies. A buffer is refilled
// only after the pass over its previous group has read it (an event per
// buffer). Each group's kept positions (and, on request, its kept K and V
// rows) go back to host memory on `stream` right after its pass. One
// cudaMemcpyAsync (or cudaMemcpy2DAsync for the window queries, one row per
// request) per copy; the library allocates no device memory.
#include <string.h>

#include <algorithm>

#include "jacap.h"
#include "jacap_dev.cuh"
#include "jacap_internal.h"

using namespace jacap;

namespace {

constexpr size_t HB_ALIGN = 1024;
inline size_t hb_align(size_t x) { return (x + HB_ALIGN - 1) & ~(HB_ALIGN - 1); }

// Sections of the caller's device buffer.
struct HostCarve {
  size_t cu, slots, kb[2], vb[2], qb[2], ws, scores, idx, kept, kout, vout, total;
  size_t ws_bytes;
};

int groups_of(const jacap_layout* L, int gl) { return (L->num_layers + gl - 1) / gl; }

// The layout of one group of `n` layers in the device buffers (dense).
jacap_layout group_layout(const jacap_layout* L, int n, const int32_t* cu_dev) {
  jacap_layout g = *L;
  g.cu_seqlens = cu_dev;
  g.num_layers = n;
  g.kv_stride_token = D;
  g.kv_stride_head = L->total_tokens * D;
  g.kv_stride_layer = (int64_t)L->num_kv_heads * L->total_tokens * D;
  g.q_stride_pos = D;
  g.q_stride_head = (int64_t)L->window * D;
  g.q_stride_layer = (int64_t)L->num_q_heads * L->window * D;
  g.q_stride_seq = (int64_t)n * g.q_stride_layer;
  return g;
}

// Host arrays must be dense: K, V [L][Hkv][N_tot][128], Q window
// [S][L][Hq][w][128]. Returns JACAP_OK or JACAP_ERR_INVALID_ARG.
jacap_status check_dense(const jacap_layout* L) {
  const int64_t kv_head = L->total_tokens * D, kv_layer = (int64_t)L->num_kv_heads * kv_head;
  const int64_t q_head = (int64_t)L->window * D, q_layer = (int64_t)L->num_q_heads * q_head,
                q_seq = (int64_t)L->num_layers * q_layer;
  if (L->kv_stride_token != D || L->kv_stride_head != kv_head || L->kv_stride_layer != kv_layer) return JACAP_ERR_INVALID_ARG;
  if (L->q_stride_pos != D || L->q_stride_head != q_head || L->q_stride_layer != q_layer || L->q_stride_seq != q_seq)
    return JACAP_ERR_INVALID_ARG;
  return JACAP_OK;
}

// Carves the device buffer; ws_bytes == 0 when the group layout is invalid.
HostCarve host_carve(const jacap_layout* L, int32_t budget, int gl, bool rows) {
  HostCarve c;
  memset(&c, 0, sizeof(c));
  const size_t es = L->dtype == JACAP_BF16 ? 2 : 4;
  const int n = std::min(gl, L->num_layers);
  const size_t S = (size_t)L->num_seqs, Hkv = (size_t)L->num_kv_heads, N = (size_t)L->total_tokens;
  const size_t kv_group = (size_t)n * Hkv * N * D * es;
  const size_t q_group = S * n * L->num_q_heads * (size_t)L->window * D * es;
  jacap_layout g = group_layout(L, n, nullptr);
  g.cu_seqlens = (const int32_t*)(uintptr_t)HB_ALIGN;  // any non-null pointer: only the size is asked
  c.ws_bytes = jacap_workspace_size(&g, budget);
  size_t o = 0;
  c.cu = o; o = hb_align(o + (S + 1) * 4);
  c.slots = o; o = hb_align(o + (size_t)groups_of(L, gl) * 4);
  for (int b = 0; b < 2; ++b) {
    c.kb[b] = o; o = hb_align(o + kv_group);
    c.vb[b] = o; o = hb_align(o + kv_group);
    c.qb[b] = o; o = hb_align(o + q_group);
  }
  c.ws = o; o = hb_align(o + c.ws_bytes);
  c.scores = o; o = hb_align(o + (size_t)n * Hkv * N * 4);
  c.idx = o; o = hb_align(o + (size_t)n * Hkv * S * budget * 4);
  c.kept = o; o = hb_align(o + S * 4);
  if (rows) {
    c.kout = o; o = hb_align(o + (size_t)n * Hkv * S * budget * D * es);
    c.vout = o; o = hb_align(o + (size_t)n * Hkv * S * budget * D * es);
  }
  c.total = o;
  return c;
}

jacap_status map_err(cudaError_t e) { return e == cudaSuccess ? JACAP_OK : JACAP_ERR_CUDA; }

}  // namespace

extern "C" {

size_t jacap_host_buffer_size(const jacap_layout* layout, int32_t budget, int32_t group_layers, int32_t copy_rows) {
  if (layout == nullptr || budget < 1 || group_layers < 1 || (copy_rows != 0 && copy_rows != 1)) return 0;
  if (layout->cu_seqlens == nullptr) return 0;
  jacap_layout probe = *layout;
  if (jacap_workspace_size(&probe, budget) == 0 || check_dense(layout) != JACAP_OK) return 0;
  const HostCarve c = host_carve(layout, budget, group_layers, copy_rows != 0);
  return c.ws_bytes == 0 ? 0 : c.total;
}

jacap_status jacap_evict_host(const jacap_layout* layout, const jacap_params* params, int32_t budget,
                              int32_t group_layers, const void* q_win_host, const void* k_host, const void* v_host,
                              const float* out_factor, int32_t* idx_host, int32_t* kept_host, void* k_out_host,
                              void* v_out_host, void* dev_buf, size_t dev_bytes, void* stream, void* copy_stream) {
  if (layout == nullptr || params == nullptr || q_win_host == nullptr || k_host == nullptr || v_host == nullptr ||
      idx_host == nullptr || kept_host == nullptr || dev_buf == nullptr || budget < 1 || group_layers < 1)
    return JACAP_ERR_INVALID_ARG;
  if ((k_out_host == nullptr) != (v_out_host == nullptr)) return JACAP_ERR_INVALID_ARG;
  const bool rows = k_out_host != nullptr;
  const size_t need = jacap_host_buffer_size(layout, budget, group_layers, rows ? 1 : 0);
  if (need == 0) {
    // report the layout's own problem the way the other entry points do
    jacap_layout probe = *layout;
    if (jacap_workspace_size(&probe, budget) == 0) {
      const jacap_status st = jacap_select(&probe, nullptr, budget, nullptr, nullptr, nullptr, 0, nullptr);
      return st == JACAP_OK ? JACAP_ERR_INVALID_ARG : st;
    }
    return JACAP_ERR_INVALID_ARG;
  }
  if (((uintptr_t)dev_buf & 1023u) != 0 || dev_bytes < need) return JACAP_ERR_WORKSPACE;
  if (out_factor != nullptr && ((uintptr_t)out_factor & 15u) != 0) return JACAP_ERR_INVALID_ARG;

  const int gl = std::min<int>(group_layers, layout->num_layers);
  const int ngroups = groups_of(layout, gl);
  const HostCarve c = host_carve(layout, budget, gl, rows);
  uint8_t* base = (uint8_t*)dev_buf;
  int32_t* cu_dev = (int32_t*)(base + c.cu);
  uint32_t* slots = (uint32_t*)(base + c.slots);
  const cudaStream_t s = (cudaStream_t)stream;
  const cudaStream_t cs = (copy_stream != nullptr && copy_stream != stream) ? (cudaStream_t)copy_stream : s;
  const bool two = cs != s;

  const size_t es = layout->dtype == JACAP_BF16 ? 2 : 4;
  const size_t S = (size_t)layout->num_seqs, Hkv = (size_t)layout->num_kv_heads, N = (size_t)layout->total_tokens;
  const size_t kv_layer = Hkv * N * D * es;                                  // bytes per layer of K (or V)
  const size_t q_layer = (size_t)layout->num_q_heads * layout->window * D * es;  // per (request, layer)
  const size_t idx_layer = Hkv * S * budget * 4, row_layer = Hkv * S * budget * D * es;

  cudaEvent_t ready[2] = {nullptr, nullptr}, freed[2] = {nullptr, nullptr};
  jacap_status st = JACAP_OK;
  auto cleanup = [&]() {
    for (int b = 0; b < 2; ++b) {
      if (ready[b] != nullptr) cudaEventDestroy(ready[b]);
      if (freed[b] != nullptr) cudaEventDestroy(freed[b]);
    }
  };
  if (two)
    for (int b = 0; b < 2 && st == JACAP_OK; ++b)
      if (cudaEventCreateWithFlags(&ready[b], cudaEventDisableTiming) != cudaSuccess ||
          cudaEventCreateWithFlags(&freed[b], cudaEventDisableTiming) != cudaSuccess)
        st = JACAP_ERR_CUDA;
  if (st == JACAP_OK)
    st = map_err(cudaMemcpyAsync(cu_dev, layout->cu_seqlens, (S + 1) * 4, cudaMemcpyHostToDevice, s));
  if (st == JACAP_OK) st = map_err(cudaMemsetAsync(slots, 0, (size_t)ngroups * 4, s));
  // the copy stream starts after the request offsets (and the slots) are in place
  if (st == JACAP_OK && two) {
    st = map_err(cudaEventRecord(freed[1], s));
    if (st == JACAP_OK) st = map_err(cudaStreamWaitEvent(cs, freed[1], 0));
  }

  for (int g = 0; g < ngroups && st == JACAP_OK; ++g) {
    const int l0 = g * gl, n = std::min(gl, layout->num_layers - l0), b = g & 1;
    uint8_t* kb = base + c.kb[b];
    uint8_t* vb = base + c.vb[b];
    uint8_t* qb = base + c.qb[b];
    // ---- host -> device copies of the group on the copy stream
    if (two && g >= 2 && (st = map_err(cudaStreamWaitEvent(cs, freed[b], 0))) != JACAP_OK) break;
    if ((st = map_err(cudaMemcpyAsync(kb, (const uint8_t*)k_host + l0 * kv_layer, n * kv_layer,
                                      cudaMemcpyHostToDevice, cs))) != JACAP_OK ||
        (st = map_err(cudaMemcpyAsync(vb, (const uint8_t*)v_host + l0 * kv_layer, n * kv_layer,
                                      cudaMemcpyHostToDevice, cs))) != JACAP_OK ||
        // request s's layers l0 .. l0 + n - 1 of the window are one row of the copy
        (st = map_err(cudaMemcpy2DAsync(qb, n * q_layer, (const uint8_t*)q_win_host + l0 * q_layer,
                                        layout->num_layers * q_layer, n * q_layer, S, cudaMemcpyHostToDevice,
                                        cs))) != JACAP_OK)
      break;
    if (two && ((st = map_err(cudaEventRecord(ready[b], cs))) != JACAP_OK ||
                (st = map_err(cudaStreamWaitEvent(s, ready[b], 0))) != JACAP_OK))
      break;
    // ---- the pass over the group on the compute stream
    const jacap_layout lg = group_layout(layout, n, cu_dev);
    void* ws = base + c.ws;
    float* scores = (float*)(base + c.scores);
    int32_t* idx = (int32_t*)(base + c.idx);
    int32_t* kept = (int32_t*)(base + c.kept);
    const float* of = out_factor == nullptr ? nullptr : out_factor + (size_t)l0 * Hkv * D * D;
    if ((st = jacap_score_out(&lg, params, qb, kb, vb, of, scores, ws, c.ws_bytes, s, nullptr, 0)) != JACAP_OK) break;
    st = rows ? jacap_select_compact(&lg, scores, budget, idx, kept, kb, vb, base + c.kout, base + c.vout, ws,
                                     c.ws_bytes, s)
              : jacap_select(&lg, scores, budget, idx, kept, ws, c.ws_bytes, s);
    if (st != JACAP_OK) break;
    if (two && (st = map_err(cudaEventRecord(freed[b], s))) != JACAP_OK) break;
    // ---- the group's status word and results back, in order on the compute stream
    if ((st = map_err(cudaMemcpyAsync(slots + g, ws, 4, cudaMemcpyDeviceToDevice, s))) != JACAP_OK ||
        (st = map_err(cudaMemcpyAsync((uint8_t*)idx_host + l0 * idx_layer, idx, n * idx_layer,
                                      cudaMemcpyDeviceToHost, s))) != JACAP_OK)
      break;
    if (rows && ((st = map_err(cudaMemcpyAsync((uint8_t*)k_out_host + l0 * row_layer, base + c.kout, n * row_layer,
                                               cudaMemcpyDeviceToHost, s))) != JACAP_OK ||
                 (st = map_err(cudaMemcpyAsync((uint8_t*)v_out_host + l0 * row_layer, base + c.vout, n * row_layer,
                                               cudaMemcpyDeviceToHost, s))) != JACAP_OK))
      break;
    if (g == ngroups - 1)
      st = map_err(cudaMemcpyAsync(kept_host, kept, S * 4, cudaMemcpyDeviceToHost, s));
  }
  // every copy and kernel enqueued above completes before the call returns
  const cudaError_t e1 = cudaStreamSynchronize(s);
  const cudaError_t e2 = two ? cudaStreamSynchronize(cs) : cudaSuccess;
  cleanup();
  if (st != JACAP_OK) return st;
  if (e1 != cudaSuccess || e2 != cudaSuccess) return JACAP_ERR_CUDA;
  // the first group whose pass reported a problem decides the status
  for (int g = 0; g < ngroups; ++g) {
    const jacap_status gs = jacap_device_status(slots + g, stream);
    if (gs != JACAP_OK) return gs;
  }
  return JACAP_OK;
}

}  // extern "C"
