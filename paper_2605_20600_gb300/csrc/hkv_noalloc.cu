// hkv_decode_attention_noalloc: decode attention that needs no workspace
// from its caller.
//
// Some callers cannot hand us device memory for scratch: a plain C host
// program with no device allocator of its own, a plugin inside a host
// framework that owns and budgets all device memory, or code on a path where
// an allocation is not allowed (for instance because it would synchronise the
// device in a latency-critical loop). For them the split-K partial results
// and the records of split heads live in one file-scope device array of
// fixed size, which every GPU that loads this library holds until the process
// exits.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <stdlib.h>
#include <string.h>

#include <mutex>

#include "hkv.h"
#include "hkv_kernels.h"

namespace {

using namespace hkv;

// Split-K partials (per CTA boundary and per CTA, up to 1 MiB), then which
// head is split at each CTA boundary, then the control block the attention
// kernel leaves for the finishing kernel: 1.06 MiB in total. The kernels write all of it
// before reading it, so nothing in it has to start at zero.
#ifndef HKV_NOALLOC_PART_BYTES
#define HKV_NOALLOC_PART_BYTES (1u << 20)
#endif
constexpr size_t kPartBytes = HKV_NOALLOC_PART_BYTES;
constexpr size_t kRecBytes = (size_t)kAttnMaxGrid * sizeof(int4);
constexpr size_t kScratchBytes = kPartBytes + kRecBytes + 256;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;

struct NoAllocDevice {
  bool ready = false;
  unsigned char *scratch = nullptr;  // device address of g_scratch
  int sms = 0;
  int ctas[2][2] = {{0, 0}, {0, 0}};  // [dtype][D == 128]
};

NoAllocDevice g_devs[kMaxDevices];
std::mutex g_mu;

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// HKV_FAULT_INJECT=decode_attention_noalloc:<code> makes the call return
// <code> before touching the GPU, like every other entry point
hkv_status injected() {
  const char *s = getenv("HKV_FAULT_INJECT");
  static const char name[] = "decode_attention_noalloc";
  if (!s) return HKV_OK;
  const size_t n = sizeof(name) - 1;
  if (strncmp(s, name, n) == 0 && s[n] == ':') return (hkv_status)atoi(s + n + 1);
  return HKV_OK;
}

// Per-device set-up, done by the first call on each device with that device
// current: the host-side name g_scratch is only a stand-in for the array, so
// its device address is looked up here and passed to the kernel.
hkv_status setup(int D, int dtype, NoAllocDevice **out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return HKV_ERR_CUDA;
  NoAllocDevice &st = g_devs[dev];
  std::lock_guard<std::mutex> lk(g_mu);
  if (!st.ready) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || p == nullptr) return HKV_ERR_CUDA;
    if (cudaDeviceGetAttribute(&st.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return HKV_ERR_CUDA;
    st.scratch = static_cast<unsigned char *>(p);
    st.ready = true;
  }
  int &c = st.ctas[dtype == HKV_BF16 ? 1 : 0][D == 128 ? 1 : 0];
  if (c == 0) {
    int n = 0;
    if (attention_prepare(D, dtype, &n) != cudaSuccess || n <= 0) return HKV_ERR_CUDA;
    c = n;
  }
  *out = &st;
  return HKV_OK;
}

}  // namespace

extern "C" hkv_status hkv_decode_attention_noalloc(const hkv_config *cfg, const hkv_cache *cache,
                                                   int layer, const void *q, float *out,
                                                   hkv_stream_t stream) {
  const hkv_status inj = injected();
  if (inj != HKV_OK) return inj;
  const hkv_status vs = hkv_validate_config(cfg);
  if (vs != HKV_OK) return vs;
  if (!cache || !cache->k || !cache->v || !cache->off || !cache->len || !cache->err || !q ||
      !out)
    return HKV_ERR_INVALID_ARG;
  if (!aligned16(cache->k) || !aligned16(cache->v) || !aligned16(q) || !aligned16(out))
    return HKV_ERR_ALIGN;
  if (layer < 0 || layer >= cfg->n_layers) return HKV_ERR_INVALID_ARG;
  const int hpl = cfg->n_seqs * cfg->n_heads;

  NoAllocDevice *st = nullptr;
  const hkv_status ss = setup(cfg->head_dim, cfg->dtype, &st);
  if (ss != HKV_OK) return ss;
  const int ctas = st->ctas[cfg->dtype == HKV_BF16 ? 1 : 0][cfg->head_dim == 128 ? 1 : 0];

  // as many CTAs as the partial area holds (kAttnInlinePieces slots per
  // boundary and one overflow slot per CTA), at most the usual grid
  const size_t per_cta =
      (kAttnInlinePieces + 1) * (size_t)attn_part_floats(cfg->head_dim) * sizeof(float);
  int grid = st->sms * ctas;
  if (grid > kAttnMaxGrid) grid = kAttnMaxGrid;
  if ((size_t)grid * per_cta > kPartBytes) grid = (int)(kPartBytes / per_cta);

  cudaStream_t s = (cudaStream_t)stream;

  AttnArgs a = {};
  a.K = cache->k;
  a.V = cache->v;
  a.off = cache->off + (size_t)layer * hpl;
  a.len = cache->len + (size_t)layer * hpl;
  a.q = q;
  a.out = out;
  a.part = reinterpret_cast<float *>(st->scratch);
  a.over = a.part + (size_t)grid * kAttnInlinePieces * attn_part_floats(cfg->head_dim);
  a.rec = reinterpret_cast<int4 *>(st->scratch + kPartBytes);
  a.ctl = reinterpret_cast<AttnCtl *>(st->scratch + kPartBytes + kRecBytes);
  a.err = cache->err;
  a.arena_tokens = cache->capacity_tokens;
  a.nheads = hpl;
  a.qscale = (float)(1.4426950408889634 / sqrt((double)cfg->head_dim));
  return launch_attention(a, cfg->head_dim, cfg->dtype, grid, false, false, s) == cudaSuccess
             ? HKV_OK
             : HKV_ERR_CUDA;
}
