// Host side of the HeadKV C-ABI (include/hkv.h): argument validation, fault
// injection for tests, per-device launch setup, the kernel launches, and the
// state export.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <vector>

#include "hkv.h"
#include "hkv_kernels.h"

namespace {

using namespace hkv;

constexpr int kMaxDevices = 64;
constexpr size_t kMaxSmem = 227 * 1024;

// Per-device launch setup, filled on first use. Every field is written at
// most once (under g_mu) and read lock-free: atomics with acquire/release
// ordering, so a thread that sees a value also sees what was set up before
// it was published.
struct DeviceState {
  std::atomic<int> sms{0};
  std::atomic<int> attn_ctas[2][2] = {};  // [dtype][D == 128]
  std::atomic<int> step_ctas[2][2] = {};
  std::atomic<size_t> update_smem[2][2] = {};
};

DeviceState g_dev[kMaxDevices];
std::mutex g_mu;

hkv_status injected(const char *name) {
  const char *s = getenv("HKV_FAULT_INJECT");
  if (!s) return HKV_OK;
  const size_t n = strlen(name);
  if (strncmp(s, name, n) == 0 && s[n] == ':') return (hkv_status)atoi(s + n + 1);
  return HKV_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int dt_index(int dtype) { return dtype == HKV_BF16 ? 1 : 0; }
int d_index(int D) { return D == 128 ? 1 : 0; }

hkv_status cuda_status(cudaError_t e) { return e == cudaSuccess ? HKV_OK : HKV_ERR_CUDA; }

// Per-device, per-(D, dtype) launch setup (shared memory limits, occupancy);
// done on the first call that needs it, outside any stream capture.
hkv_status device_state(DeviceState **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return HKV_ERR_CUDA;
  DeviceState &st = g_dev[dev];
  if (st.sms.load(std::memory_order_acquire) == 0) {
    std::lock_guard<std::mutex> lk(g_mu);
    if (st.sms.load(std::memory_order_relaxed) == 0) {
      int n = 0;
      if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
        return HKV_ERR_CUDA;
      st.sms.store(n, std::memory_order_release);
    }
  }
  *out = &st;
  return HKV_OK;
}

// CTAs per SM of the decode kernels (both designs share the grid)
hkv_status attention_ctas(DeviceState *st, int D, int dtype, int *ctas) {
  std::atomic<int> &c = st->attn_ctas[dt_index(dtype)][d_index(D)];
  int v = c.load(std::memory_order_acquire);
  if (v == 0) {
    std::lock_guard<std::mutex> lk(g_mu);
    v = c.load(std::memory_order_relaxed);
    if (v == 0) {
      int n = 0;
      if (attention_prepare(D, dtype, &n) != cudaSuccess || n <= 0) return HKV_ERR_CUDA;
      v = n;
      c.store(v, std::memory_order_release);
    }
  }
  *ctas = v;
  return HKV_OK;
}

hkv_status update_ready(DeviceState *st, int D, int dtype, size_t smem) {
  std::atomic<size_t> &have = st->update_smem[dt_index(dtype)][d_index(D)];
  if (smem > kMaxSmem) return HKV_ERR_CAPACITY;
  if (have.load(std::memory_order_acquire) < smem) {
    std::lock_guard<std::mutex> lk(g_mu);
    if (have.load(std::memory_order_relaxed) < smem) {
      if (update_prepare(D, dtype, smem) != cudaSuccess) return HKV_ERR_CUDA;
      have.store(smem, std::memory_order_release);
    }
  }
  return HKV_OK;
}

hkv_status check_cache(const hkv_cache *c) {
  if (!c || !c->k || !c->v || !c->pos || !c->off || !c->cap || !c->len || !c->nbuf || !c->ntok ||
      !c->label || !c->qbuf || !c->err)
    return HKV_ERR_INVALID_ARG;
  if (!aligned16(c->k) || !aligned16(c->v) || !aligned16(c->qbuf)) return HKV_ERR_ALIGN;
  if (c->capacity_tokens <= 0) return HKV_ERR_CAPACITY;
  return HKV_OK;
}

CacheArgs cache_args(const hkv_cache *c) {
  CacheArgs a;
  a.K = c->k;
  a.V = c->v;
  a.pos = c->pos;
  a.off = c->off;
  a.cap = c->cap;
  a.len = c->len;
  a.nbuf = c->nbuf;
  a.ntok = c->ntok;
  a.label = c->label;
  a.qbuf = c->qbuf;
  a.err = c->err;
  a.arena_tokens = c->capacity_tokens;
  return a;
}

MethodArgs method_args(const hkv_config *cfg) {
  MethodArgs m;
  m.C = cfg->n_cond;
  m.w = cfg->recent_w;
  m.w_loc = cfg->local_w;
  m.P = cfg->period;
  m.r_s = cfg->r_s;
  m.tau = (float)cfg->tau;
  m.grid2d = cfg->distance_mode == HKV_DIST_GRID2D ? 1 : 0;
  m.row_len = cfg->row_len;
  return m;
}

int heads_per_layer(const hkv_config *c) { return c->n_seqs * c->n_heads; }

// longest segment any call may see: a dense head (C + E) or a compressed
// global head right before its update (C + B_g + P)
// the longest segment the config allows: the dense cache at grouping, or a
// global head's C + budget + P tokens (never more than C + N); a
// redistributed budget reaches B_g + (H - 1)(B_g - w) for a group of one
// global head
int max_segment(const hkv_config *c) {
  const int a = c->n_cond + c->group_at;
  long long bud = c->global_budget;
  if (c->budget_mode == HKV_BUDGET_REDISTRIBUTE)
    bud += (long long)(c->n_heads - 1) * (c->global_budget - c->recent_w);
  long long kept = bud + c->period;
  if (kept > c->n_image) kept = c->n_image;
  const int b = c->n_cond + (int)kept;
  return a > b ? a : b;
}

size_t align256(size_t b) { return (b + 255) & ~(size_t)255; }

constexpr size_t kCtlBytes = 256;  // AttnCtl, padded

// Workspace of the decode kernels, in this order: split-K partials
// (kAttnInlinePieces slots per CTA boundary, one overflow slot per CTA), the
// record of the head split at each CTA boundary, the control block the
// two-kernel design's attention kernel leaves for its finishing kernel, the
// epoch-tagged partial results of the one-launch step (two slots of D + 2
// 8-byte pairs per CTA) and its per-layer barrier words.
struct WsLayout {
  size_t part, over, rec, ctl, pslot, bar, total;
};

WsLayout ws_layout(const hkv_config *c) {
  WsLayout w;
  const size_t pf = attn_part_floats(c->head_dim) * sizeof(float);
  w.part = 0;
  w.over = w.part + align256((size_t)kAttnMaxGrid * kAttnInlinePieces * pf);
  w.rec = w.over + align256((size_t)kAttnMaxGrid * pf);
  w.ctl = w.rec + align256((size_t)kAttnMaxGrid * sizeof(int4));
  w.pslot = w.ctl + kCtlBytes;
  w.bar = w.pslot + align256((size_t)kAttnMaxGrid * 2 * (c->head_dim + 2) * 8);
  w.total = w.bar + align256((size_t)c->n_layers * 4 * sizeof(uint32_t));
  return w;
}

// Fills the attention launch arguments for one layer; the workspace holds
// the split-K partials (per CTA boundary, and overflow slots per CTA), which
// head is split at each CTA boundary and the control block the attention
// kernel leaves for the finishing kernel.
AttnArgs attn_args(const hkv_config *cfg, const hkv_cache *cache, int layer, const void *q,
                   float *out, void *workspace) {
  const int hpl = cfg->n_seqs * cfg->n_heads;
  AttnArgs a = {};
  a.K = cache->k;
  a.V = cache->v;
  a.off = cache->off + (size_t)layer * hpl;
  a.len = cache->len + (size_t)layer * hpl;
  a.cap = cache->cap + (size_t)layer * hpl;
  a.q = q;
  a.out = out;
  unsigned char *ws = static_cast<unsigned char *>(workspace);
  const WsLayout w = ws_layout(cfg);
  a.part = reinterpret_cast<float *>(ws + w.part);
  a.over = reinterpret_cast<float *>(ws + w.over);
  a.rec = reinterpret_cast<int4 *>(ws + w.rec);
  a.ctl = reinterpret_cast<AttnCtl *>(ws + w.ctl);
  a.pslot = reinterpret_cast<unsigned long long *>(ws + w.pslot);
  a.bar = reinterpret_cast<uint32_t *>(ws + w.bar) + (size_t)layer * 4;
  a.n_layers = cfg->n_layers;
  a.err = cache->err;
  a.pos = cache->pos;
  a.nbuf = cache->nbuf;
  a.ntok = cache->ntok;
  a.label = cache->label;
  a.qbuf = cache->qbuf;
  a.layer_base = layer * hpl;
  a.period = cfg->period;
  a.n_cond = cfg->n_cond;
  a.arena_tokens = cache->capacity_tokens;
  a.nheads = hpl;
  a.qscale = (float)(1.4426950408889634 / sqrt((double)cfg->head_dim));
  return a;
}

// CTAs per SM of the one-launch step: kStepActivePerSm, if the kernel can
// have that many resident (its own setup, once per device and shape)
hkv_status step_ctas(DeviceState *st, int D, int dtype, int *ctas) {
  std::atomic<int> &c = st->step_ctas[dt_index(dtype)][d_index(D)];
  int v = c.load(std::memory_order_acquire);
  if (v == 0) {
    std::lock_guard<std::mutex> lk(g_mu);
    v = c.load(std::memory_order_relaxed);
    if (v == 0) {
      int m = 0;
      if (step_prepare(D, dtype, &m) != cudaSuccess || m <= 0) return HKV_ERR_CUDA;
      v = m < kStepActivePerSm ? m : kStepActivePerSm;
      c.store(v, std::memory_order_release);
    }
  }
  *ctas = v;
  return HKV_OK;
}

hkv_status step_grid(const hkv_config *cfg, int *grid) {
  DeviceState *st;
  hkv_status s = device_state(&st);
  if (s != HKV_OK) return s;
  int ctas = 0;
  s = step_ctas(st, cfg->head_dim, cfg->dtype, &ctas);
  if (s != HKV_OK) return s;
  const int g = st->sms.load(std::memory_order_acquire) * ctas;
  *grid = g > kAttnMaxGrid ? kAttnMaxGrid : g;
  return HKV_OK;
}

// attention CTAs: every SM filled
hkv_status attn_grid(const hkv_config *cfg, int *grid) {
  DeviceState *st;
  hkv_status s = device_state(&st);
  if (s != HKV_OK) return s;
  int ctas = 0;
  s = attention_ctas(st, cfg->head_dim, cfg->dtype, &ctas);
  if (s != HKV_OK) return s;
  const int g = st->sms.load(std::memory_order_acquire) * ctas;
  *grid = g > kAttnMaxGrid ? kAttnMaxGrid : g;
  return HKV_OK;
}

// Whether hkv_decode_step runs as one launch (hkv_step.cu). It must fit the
// kernel's head table: a range of c tiles holds at most c + 1 heads (a head
// has at least one tile in a step, its new token), and c is at most the
// layer's tile count over the grid, bounded by every head at the longest
// segment the config allows. Where it fits, one launch is the faster design
// on every model shape measured (each shape A/B in one process on GB300).
// HKV_STEP_TWO_KERNELS in the environment forces the two-kernel design
// (tests of both).
bool one_launch_step(const hkv_config *cfg, int grid) {
  if (getenv("HKV_STEP_TWO_KERNELS")) return false;
  const long long tt = step_tile_rows(cfg->head_dim, cfg->dtype);
  const long long tiles = (long long)heads_per_layer(cfg) * ((max_segment(cfg) + tt - 1) / tt);
  long long chunk = (tiles + grid - 1) / grid;
  if (chunk < 2) chunk = 2;
  return chunk + 1 <= kStepTable;
}

#define HKV_TRY(x)                 \
  do {                             \
    hkv_status s_ = (x);           \
    if (s_ != HKV_OK) return s_;   \
  } while (0)

}  // namespace

extern "C" {

const char *hkv_status_str(hkv_status s) {
  switch (s) {
    case HKV_OK: return "ok";
    case HKV_ERR_INVALID_ARG: return "invalid argument";
    case HKV_ERR_SHAPE: return "unsupported shape";
    case HKV_ERR_CAPACITY: return "capacity exceeded";
    case HKV_ERR_STATE: return "cache in the wrong state";
    case HKV_ERR_BOUNDS: return "segment outside the arena";
    case HKV_ERR_TIMEOUT: return "device wait timed out";
    case HKV_ERR_CUDA: return "CUDA error";
    case HKV_ERR_ALIGN: return "pointer not 16-byte aligned";
  }
  return "unknown status";
}

hkv_status hkv_validate_config(const hkv_config *c) {
  HKV_TRY(injected("validate_config"));
  if (!c) return HKV_ERR_INVALID_ARG;
  if (c->dtype != HKV_FP32 && c->dtype != HKV_BF16) return HKV_ERR_INVALID_ARG;
  if (c->head_dim != 64 && c->head_dim != 128) return HKV_ERR_SHAPE;
  if (c->n_layers <= 0 || c->n_seqs <= 0 || c->n_heads <= 0 || c->n_cond < 0 ||
      c->n_image <= 0 || c->row_len <= 0 || c->recent_w <= 0 || c->local_w <= 0 ||
      c->period <= 0 || c->group_at <= 0)
    return HKV_ERR_SHAPE;
  if (c->period > c->group_at || c->group_at > c->n_image) return HKV_ERR_SHAPE;
  if (c->global_budget < c->recent_w || c->global_budget > c->n_image) return HKV_ERR_SHAPE;
  if ((long long)c->n_layers * c->n_seqs * c->n_heads > (1ll << 30)) return HKV_ERR_SHAPE;
  if ((long long)c->n_cond + c->n_image + c->period > (1ll << 24)) return HKV_ERR_SHAPE;
  if (!(c->tau > 0.0 && c->tau <= 1.0) || !(c->r_s >= 0.0 && c->r_s <= 1.0))
    return HKV_ERR_INVALID_ARG;
  if (c->budget_mode != HKV_BUDGET_PAPER && c->budget_mode != HKV_BUDGET_REDISTRIBUTE)
    return HKV_ERR_INVALID_ARG;
  if ((c->distance_mode != HKV_DIST_RASTER && c->distance_mode != HKV_DIST_GRID2D) ||
      c->reserved != 0)
    return HKV_ERR_INVALID_ARG;
  if (c->distance_mode == HKV_DIST_GRID2D) {  // squared grid distances fit 31 bits
    const long long rows = (c->n_image + c->row_len - 1) / c->row_len;
    if ((rows - 1) * (rows - 1) + (long long)(c->row_len - 1) * (c->row_len - 1) >= (1ll << 31))
      return HKV_ERR_SHAPE;
  }
  // a capacity (C + budget + P) stays an int32
  if ((long long)c->n_cond + (long long)c->n_heads * c->global_budget + c->period > 0x7fffffffLL)
    return HKV_ERR_SHAPE;
  return HKV_OK;
}

hkv_status hkv_global_budget(int64_t rho_num, int64_t rho_den, int32_t n_image,
                             int32_t *budget_out) {
  HKV_TRY(injected("global_budget"));
  if (!budget_out) return HKV_ERR_INVALID_ARG;
  if (rho_num <= 0 || rho_den <= 0 || rho_num > rho_den || rho_den > 0x7fffffffLL ||
      n_image <= 0)
    return HKV_ERR_INVALID_ARG;
  // Sec. 5.1: rho * N image tokens, rounded down; exact (num * N < 2^62)
  *budget_out = (int32_t)(rho_num * (int64_t)n_image / rho_den);
  return HKV_OK;
}

hkv_status hkv_update_due(const hkv_config *cfg, int32_t t, int32_t *due_out) {
  HKV_TRY(injected("update_due"));
  HKV_TRY(hkv_validate_config(cfg));
  if (!due_out || t < 0) return HKV_ERR_INVALID_ARG;
  // Sec. 4, Efficient Cache Update: the grouping step (image token E - 1)
  // runs the first update; after it the buffer fills every P tokens, and the
  // update that empties it runs before the step of the token after the P-th
  const int E = cfg->group_at, P = cfg->period;
  *due_out = t > E && (t - E) % P == 0 ? 1 : 0;
  return HKV_OK;
}

size_t hkv_workspace_size(const hkv_config *c) {
  if (!c || hkv_validate_config(c) != HKV_OK) return 0;
  return ws_layout(c).total;
}

hkv_status hkv_init_dense(const hkv_config *cfg, const hkv_cache *cache, hkv_stream_t stream) {
  HKV_TRY(injected("init_dense"));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(cache));
  const int seg = cfg->n_cond + cfg->group_at;
  const long long n = (long long)cfg->n_layers * heads_per_layer(cfg);
  if (cache->capacity_tokens < n * seg) return HKV_ERR_CAPACITY;
  return cuda_status(launch_init_dense(cache_args(cache), (int)n, seg, (cudaStream_t)stream));
}

hkv_status hkv_prefill(const hkv_config *cfg, const hkv_cache *cache, int layer, const void *kc,
                       const void *vc, hkv_stream_t stream) {
  HKV_TRY(injected("prefill"));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(cache));
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  if (cfg->n_cond > 0 && (!kc || !vc)) return HKV_ERR_INVALID_ARG;
  if (cfg->n_cond > 0 && (!aligned16(kc) || !aligned16(vc))) return HKV_ERR_ALIGN;
  const int hpl = heads_per_layer(cfg);
  return cuda_status(launch_prefill(cache_args(cache), layer * hpl, hpl, cfg->n_cond, kc, vc,
                                    cfg->head_dim, cfg->dtype, (cudaStream_t)stream));
}

hkv_status hkv_append_evict(const hkv_config *cfg, const hkv_cache *cache, int layer,
                            const void *q, const void *k, const void *v, hkv_stream_t stream) {
  HKV_TRY(injected("append_evict"));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(cache));
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  if (!q || !k || !v) return HKV_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v)) return HKV_ERR_ALIGN;
  DeviceState *st;
  HKV_TRY(device_state(&st));
  const size_t smem = update_smem_bytes(max_segment(cfg), cfg->head_dim, cfg->period, cfg->dtype);
  HKV_TRY(update_ready(st, cfg->head_dim, cfg->dtype, smem));
  const int hpl = heads_per_layer(cfg);
  return cuda_status(launch_append_evict(cache_args(cache), method_args(cfg), layer * hpl, hpl, q,
                                         k, v, cfg->head_dim, cfg->dtype, smem,
                                         (cudaStream_t)stream));
}

hkv_status hkv_decode_attention(const hkv_config *cfg, const hkv_cache *cache, int layer,
                                const void *q, float *out, void *workspace, size_t ws_bytes,
                                hkv_stream_t stream) {
  HKV_TRY(injected("decode_attention"));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(cache));
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  if (!q || !out || !workspace) return HKV_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out) || !aligned16(workspace)) return HKV_ERR_ALIGN;
  if (ws_bytes < hkv_workspace_size(cfg)) return HKV_ERR_CAPACITY;
  int grid = 0;
  HKV_TRY(attn_grid(cfg, &grid));
  const AttnArgs a = attn_args(cfg, cache, layer, q, out, workspace);
  return cuda_status(
      launch_attention(a, cfg->head_dim, cfg->dtype, grid, false, false, (cudaStream_t)stream));
}

namespace {

hkv_status decode_step(const char *name, const hkv_config *cfg, const hkv_cache *cache, int layer,
                       const void *q, const void *k, const void *v, float *out,
                       uint8_t *label_out, void *workspace, size_t ws_bytes, int flags,
                       hkv_stream_t stream) {
  HKV_TRY(injected(name));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(cache));
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  if (!q || !k || !v || !out || !workspace) return HKV_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out) || !aligned16(workspace))
    return HKV_ERR_ALIGN;
  if (ws_bytes < hkv_workspace_size(cfg)) return HKV_ERR_CAPACITY;
  if (flags & ~HKV_STEP_PREFETCH) return HKV_ERR_INVALID_ARG;
  int grid = 0;
  HKV_TRY(attn_grid(cfg, &grid));
  AttnArgs a = attn_args(cfg, cache, layer, q, out, workspace);
  a.k_new = k;
  a.v_new = v;
  a.prefetch = (flags & HKV_STEP_PREFETCH) ? 1 : 0;
  a.label_out = label_out;
  a.w_loc = cfg->local_w;
  a.tau = (float)cfg->tau;
  if (!label_out) {
    int sgrid = 0;
    HKV_TRY(step_grid(cfg, &sgrid));
    if (one_launch_step(cfg, sgrid))
      return cuda_status(launch_step(a, cfg->head_dim, cfg->dtype, sgrid, (cudaStream_t)stream));
  }
  return cuda_status(launch_attention(a, cfg->head_dim, cfg->dtype, grid, true,
                                      label_out != nullptr, (cudaStream_t)stream));
}

}  // namespace

hkv_status hkv_decode_step(const hkv_config *cfg, const hkv_cache *cache, int layer,
                           const void *q, const void *k, const void *v, float *out,
                           void *workspace, size_t ws_bytes, int flags, hkv_stream_t stream) {
  return decode_step("decode_step", cfg, cache, layer, q, k, v, out, nullptr, workspace, ws_bytes,
                     flags, stream);
}

int hkv_decode_step_launches(const hkv_config *cfg) {
  if (hkv_validate_config(cfg) != HKV_OK) return 0;
  int grid = 0;
  if (step_grid(cfg, &grid) != HKV_OK) return 0;
  return one_launch_step(cfg, grid) ? 1 : 2;
}

hkv_status hkv_decode_step_identify(const hkv_config *cfg, const hkv_cache *cache, int layer,
                                    const void *q, const void *k, const void *v, float *out,
                                    uint8_t *label_out, void *workspace, size_t ws_bytes,
                                    int flags, hkv_stream_t stream) {
  if (!label_out) return HKV_ERR_INVALID_ARG;
  // the fused count is the raster one (the newest rows of the segment)
  if (cfg && cfg->distance_mode != HKV_DIST_RASTER) return HKV_ERR_INVALID_ARG;
  return decode_step("decode_step_identify", cfg, cache, layer, q, k, v, out, label_out,
                     workspace, ws_bytes, flags, stream);
}

namespace {

// the periodic update of the layers [first, first + count) in one launch
hkv_status evict_layers(const hkv_config *cfg, const hkv_cache *cache, int first, int count,
                        hkv_stream_t stream) {
  DeviceState *st;
  HKV_TRY(device_state(&st));
  const size_t smem = update_smem_bytes(max_segment(cfg), cfg->head_dim, cfg->period, cfg->dtype);
  HKV_TRY(update_ready(st, cfg->head_dim, cfg->dtype, smem));
  const long long hpl = heads_per_layer(cfg);
  if (hpl * count > 0x7FFFFFFFLL) return HKV_ERR_SHAPE;  // one CTA per head
  return cuda_status(launch_evict(cache_args(cache), method_args(cfg), (int)(first * hpl),
                                  (int)(count * hpl), cfg->head_dim, cfg->dtype, smem,
                                  (cudaStream_t)stream));
}

}  // namespace

hkv_status hkv_evict(const hkv_config *cfg, const hkv_cache *cache, int layer,
                     hkv_stream_t stream) {
  HKV_TRY(injected("evict"));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(cache));
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  return evict_layers(cfg, cache, layer, 1, stream);
}

hkv_status hkv_evict_all(const hkv_config *cfg, const hkv_cache *cache, hkv_stream_t stream) {
  HKV_TRY(injected("evict_all"));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(cache));
  return evict_layers(cfg, cache, 0, cfg->n_layers, stream);
}

hkv_status hkv_identify_heads(const hkv_config *cfg, const hkv_cache *cache, int layer,
                              const void *q, uint8_t *label_out, int32_t *nh_out,
                              hkv_stream_t stream) {
  HKV_TRY(injected("identify_heads"));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(cache));
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  if (!q || !label_out) return HKV_ERR_INVALID_ARG;
  if (!aligned16(q)) return HKV_ERR_ALIGN;
  DeviceState *st;
  HKV_TRY(device_state(&st));
  const int max_len = cfg->n_cond + cfg->group_at;
  const size_t upd = update_smem_bytes(max_segment(cfg), cfg->head_dim, cfg->period, cfg->dtype);
  const size_t need = identify_smem_bytes(max_len, cfg->period,
                                          cfg->distance_mode == HKV_DIST_GRID2D, false);
  HKV_TRY(update_ready(st, cfg->head_dim, cfg->dtype, upd > need ? upd : need));
  const int hpl = heads_per_layer(cfg);
  return cuda_status(launch_identify(cache_args(cache), method_args(cfg), layer * hpl, hpl, q,
                                     label_out, nh_out, cfg->head_dim, cfg->dtype, max_len,
                                     (cudaStream_t)stream));
}

hkv_status hkv_identify_heads_multi(const hkv_config *cfg, const hkv_cache *cache, int layer,
                                    uint8_t *label_out, int32_t *nh_out, hkv_stream_t stream) {
  HKV_TRY(injected("identify_heads_multi"));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(cache));
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  if (!label_out) return HKV_ERR_INVALID_ARG;
  DeviceState *st;
  HKV_TRY(device_state(&st));
  const int max_len = cfg->n_cond + cfg->group_at;
  const size_t upd = update_smem_bytes(max_segment(cfg), cfg->head_dim, cfg->period, cfg->dtype);
  const size_t need = identify_smem_bytes(max_len, cfg->period,
                                          cfg->distance_mode == HKV_DIST_GRID2D, true);
  HKV_TRY(update_ready(st, cfg->head_dim, cfg->dtype, upd > need ? upd : need));
  const int hpl = heads_per_layer(cfg);
  return cuda_status(launch_identify_multi(cache_args(cache), method_args(cfg), layer * hpl, hpl,
                                           label_out, nh_out, cfg->head_dim, cfg->dtype, max_len,
                                           (cudaStream_t)stream));
}

hkv_status hkv_allocate_budgets(const hkv_config *cfg, const uint8_t *label, int32_t *budget,
                                int32_t *cap, int64_t *off, int64_t *total_tokens,
                                hkv_stream_t stream) {
  HKV_TRY(injected("allocate_budgets"));
  HKV_TRY(hkv_validate_config(cfg));
  if (!label || !budget || !cap || !off || !total_tokens) return HKV_ERR_INVALID_ARG;
  const int n = cfg->n_layers * heads_per_layer(cfg);
  cudaStream_t s = (cudaStream_t)stream;
  if (launch_budgets(label, budget, cap, off, n, cfg->n_cond, cfg->global_budget, cfg->recent_w,
                     cfg->period,
                     cfg->budget_mode == HKV_BUDGET_REDISTRIBUTE ? cfg->n_heads : 0,
                     s) != cudaSuccess)
    return HKV_ERR_CUDA;
  int64_t last_off = 0;
  int32_t last_cap = 0;
  if (cudaMemcpyAsync(&last_off, off + (n - 1), sizeof(last_off), cudaMemcpyDeviceToHost, s) !=
          cudaSuccess ||
      cudaMemcpyAsync(&last_cap, cap + (n - 1), sizeof(last_cap), cudaMemcpyDeviceToHost, s) !=
          cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return HKV_ERR_CUDA;
  if (last_off < 0) return HKV_ERR_STATE;
  *total_tokens = last_off + last_cap;
  return HKV_OK;
}

hkv_status hkv_repack(const hkv_config *cfg, const hkv_cache *dense, const hkv_cache *ragged,
                      int layer, hkv_stream_t stream) {
  HKV_TRY(injected("repack"));
  HKV_TRY(hkv_validate_config(cfg));
  HKV_TRY(check_cache(dense));
  HKV_TRY(check_cache(ragged));
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  if (dense->qbuf != ragged->qbuf) return HKV_ERR_INVALID_ARG;
  DeviceState *st;
  HKV_TRY(device_state(&st));
  const size_t smem = update_smem_bytes(max_segment(cfg), cfg->head_dim, cfg->period, cfg->dtype);
  HKV_TRY(update_ready(st, cfg->head_dim, cfg->dtype, smem));
  const int hpl = heads_per_layer(cfg);
  return cuda_status(launch_repack(cache_args(dense), cache_args(ragged), method_args(cfg),
                                   layer * hpl, hpl, cfg->head_dim, cfg->dtype, smem,
                                   (cudaStream_t)stream));
}

hkv_status hkv_export_state(const hkv_config *cfg, const hkv_cache *cache, int layer,
                            uint8_t *label_out, int32_t *len_out, int32_t *nbuf_out,
                            int32_t *ntok_out, int32_t *pos_out, int64_t pos_capacity,
                            int64_t *pos_count, hkv_stream_t stream) {
  HKV_TRY(injected("export_state"));
  HKV_TRY(hkv_validate_config(cfg));
  if (!cache || !cache->off || !cache->len || !cache->nbuf || !cache->ntok || !cache->label ||
      (pos_out && !cache->pos) || pos_capacity < 0)
    return HKV_ERR_INVALID_ARG;
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  const int hpl = heads_per_layer(cfg);
  const size_t base = (size_t)layer * hpl;
  cudaStream_t s = (cudaStream_t)stream;
  std::vector<int64_t> off(hpl);
  std::vector<int32_t> len(hpl);
  auto d2h = [&](void *dst, const void *src, size_t bytes) {
    return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToHost, s) == cudaSuccess;
  };
  bool ok = d2h(off.data(), cache->off + base, hpl * sizeof(int64_t)) &&
            d2h(len.data(), cache->len + base, hpl * sizeof(int32_t));
  if (label_out) ok = ok && d2h(label_out, cache->label + base, hpl * sizeof(uint8_t));
  if (nbuf_out) ok = ok && d2h(nbuf_out, cache->nbuf + base, hpl * sizeof(int32_t));
  if (ntok_out) ok = ok && d2h(ntok_out, cache->ntok + base, hpl * sizeof(int32_t));
  if (!ok || cudaStreamSynchronize(s) != cudaSuccess) return HKV_ERR_CUDA;
  if (len_out) std::copy(len.begin(), len.end(), len_out);
  int64_t total = 0, lo = INT64_MAX, hi = 0;
  for (int h = 0; h < hpl; ++h) {
    if (len[h] < 0 || off[h] < 0 || off[h] + len[h] > cache->capacity_tokens) return HKV_ERR_BOUNDS;
    total += len[h];
    if (len[h] > 0) {
      lo = std::min(lo, off[h]);
      hi = std::max(hi, off[h] + (int64_t)len[h]);
    }
  }
  if (pos_count) *pos_count = total;
  if (!pos_out || total == 0) return HKV_OK;
  if (pos_capacity < total) return HKV_ERR_CAPACITY;
  // one copy of the span the layer's live tokens occupy, then packed
  std::vector<int32_t> span((size_t)(hi - lo));
  if (!d2h(span.data(), cache->pos + lo, span.size() * sizeof(int32_t)) ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return HKV_ERR_CUDA;
  int64_t w = 0;
  for (int h = 0; h < hpl; ++h)
    for (int j = 0; j < len[h]; ++j) pos_out[w++] = span[(size_t)(off[h] - lo + j)];
  return HKV_OK;
}

hkv_status hkv_check(const hkv_cache *cache, hkv_stream_t stream) {
  HKV_TRY(injected("check"));
  if (!cache || !cache->err) return HKV_ERR_INVALID_ARG;
  cudaStream_t s = (cudaStream_t)stream;
  uint32_t word = 0;
  if (cudaMemcpyAsync(&word, cache->err, sizeof(word), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return HKV_ERR_CUDA;
  return (hkv_status)word;
}

}  // extern "C"
