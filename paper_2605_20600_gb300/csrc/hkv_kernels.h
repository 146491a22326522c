// Host-side launchers of the HeadKV kernels (internal to libheadkv.so).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "hkv.h"

namespace hkv {

// Written by block 0 of the attention kernel for the finishing kernel.
struct AttnCtl {
  int valid;         // 1: the attention launch passed its checks
  int pad[3];
};

// Split-K decode attention over one layer of a ragged cache, optionally
// fused with the append of the step's new token: an attention kernel that
// streams the cache and a finishing kernel that combines split heads,
// appends the new token and advances the counters.
struct AttnArgs {
  void *K, *V;                // arena
  const int64_t *off;         // layer slice of segment offsets
  int32_t *len;               // layer slice of live lengths
  const int32_t *cap;         // layer slice of capacities (fused)
  const void *q;              // [nheads][D]
  const void *k_new, *v_new;  // [nheads][D] new token (fused)
  float *out;                 // [nheads][D]
  // Partial results (attn_part_floats(D) floats each) of heads split over
  // several CTA ranges. The head split at CTA boundary k (its first row in
  // CTA k - 1's range, pieces in CTAs k - 1 .. k + np - 2) keeps pieces
  // j < kAttnInlinePieces in part[k][j] and the others in over[k - 1 + j],
  // the slot of the CTA that computed them.
  float *part;                // [grid][kAttnInlinePieces][...]
  float *over;                // [grid][...]
  // For each CTA k >= 1 whose range starts inside a head whose first row
  // lies in CTA k - 1's range: {head, np, 0, 0}; else {-1, 0, 0, 0}.
  // Written by every launch before the finishing kernel reads it.
  int4 *rec;                  // [grid]
  int grid;                   // attention CTAs (set by launch_attention)
  AttnCtl *ctl;
  uint32_t *err;
  // fused append: full [L*S*H] arrays and the layer's first flat head
  int32_t *pos, *nbuf, *ntok;
  const uint8_t *label;
  void *qbuf;
  int layer_base;
  int period, n_cond;
  int64_t arena_tokens;
  int nheads;
  float qscale;               // log2(e) / sqrt(D)
  int prefetch;               // read the layer's cache before waiting for the
                              // previous kernel (its writes do not touch it)
  // identification fused into the step (Sec. 4, Step 2): a head is local iff
  // its newest w_loc - 1 tokens hold at least tau of its attention
  uint8_t *label_out;         // [L*S*H]
  int w_loc;
  float tau;
  // one-launch step (hkv_step.cu): the layer's barrier words {arrivals,
  // generation, worst status of a bad step, unused}, the arrivals and the
  // status zero between launches; the partial results of split heads
  // as (value, launch epoch) pairs, two slots per CTA (the piece at the end
  // of its range, the piece at its start), [grid][2][D + 2]
  uint32_t *bar;
  unsigned long long *pslot;
  int n_layers;
};

// decode attention CTAs: one producer warp (TMA), consumer warps, one
// epilogue warp (merges, outputs, partial results); at most kAttnMaxGrid
constexpr int kAttnMaxGrid = 4096;
// finishing kernel: CTAs of two warps, each warp for 32 heads' counters and
// one CTA boundary's split head; at 64 registers a thread, two such CTAs fit
// on an SM beside two attention CTAs (measured: one-warp CTAs 1 % slower,
// four-warp CTAs, one per SM, 10 % slower)
#ifndef HKV_FINISH_THREADS
#define HKV_FINISH_THREADS 64
#endif
constexpr int kFinishThreads = HKV_FINISH_THREADS;
constexpr int kFinishRegs = 64;
// floats of one split-K partial result: D accumulators, the running maximum
// and the sum, padded to 16 bytes for vector access
__host__ __device__ constexpr int attn_part_floats(int D) { return D + 4; }
// pieces of a split head kept per CTA boundary (loaded with its record)
constexpr int kAttnInlinePieces = 4;

// one-launch decode step: heads of a CTA's range it keeps in shared memory
#ifndef HKV_STEP_TABLE
#define HKV_STEP_TABLE 128
#endif
constexpr int kStepTable = HKV_STEP_TABLE;

size_t attention_smem_bytes(int D, int dtype);
// rows of K (and of V) per pipeline stage of the one-launch step
int step_tile_rows(int D, int dtype);
// CTAs per SM of the one-launch step's grid, and the shared memory and
// occupancy setup of its kernel (resident CTAs per SM)
#ifndef HKV_STEP_ACTIVE_PER_SM
#define HKV_STEP_ACTIVE_PER_SM 2
#endif
constexpr int kStepActivePerSm = HKV_STEP_ACTIVE_PER_SM;

cudaError_t step_prepare(int D, int dtype, int *ctas_per_sm);
// the fused decode step of one layer in one launch (append + attention,
// merges of split heads and counters in the same kernel); `grid` CTAs, at
// most kAttnMaxGrid, a CTA's range spanning at most kStepTable heads
cudaError_t launch_step(const AttnArgs &a, int D, int dtype, int grid, cudaStream_t s);
cudaError_t attention_prepare(int D, int dtype, int *ctas_per_sm);
// launches the attention kernel on `grid` CTAs (at most kAttnMaxGrid) and the
// finishing kernel behind it; identify (fused only): also the Step 2 label of
// every head into label_out
cudaError_t launch_attention(const AttnArgs &a, int D, int dtype, int grid, bool fused,
                             bool identify, cudaStream_t s);

// per-head cache maintenance (append / update / repack / prefill / identify)
struct CacheArgs {
  void *K, *V;
  int32_t *pos;
  const int64_t *off;
  const int32_t *cap;
  int32_t *len, *nbuf, *ntok;
  const uint8_t *label;
  void *qbuf;
  uint32_t *err;
  int64_t arena_tokens;
};

struct MethodArgs {
  int C, w, w_loc, P;  // a global head's history budget comes from its capacity
  double r_s;
  float tau;
  int grid2d;   // grid-distance count of Step 2 and long-range subset of Eq. 5
  int row_len;  // image tokens per grid row
};

constexpr int kCacheThreads = 256;

// dynamic shared memory of the update paths for segments of up to max_len
// tokens and a query ring of P rows
size_t update_smem_bytes(int max_len, int D, int P, int dtype);
cudaError_t update_prepare(int D, int dtype, size_t smem);

cudaError_t launch_append_evict(const CacheArgs &c, const MethodArgs &m, int layer_base,
                                int nheads, const void *q, const void *k, const void *v, int D,
                                int dtype, size_t smem, cudaStream_t s);
cudaError_t launch_evict(const CacheArgs &c, const MethodArgs &m, int layer_base, int nheads,
                         int D, int dtype, size_t smem, cudaStream_t s);
cudaError_t launch_repack(const CacheArgs &dense, const CacheArgs &ragged, const MethodArgs &m,
                          int layer_base, int nheads, int D, int dtype, size_t smem,
                          cudaStream_t s);
cudaError_t launch_prefill(const CacheArgs &c, int layer_base, int nheads, int C, const void *kc,
                           const void *vc, int D, int dtype, cudaStream_t s);
cudaError_t launch_init_dense(const CacheArgs &c, int nheads_total, int seg_tokens,
                              cudaStream_t s);
cudaError_t launch_identify(const CacheArgs &c, const MethodArgs &m, int layer_base, int nheads,
                            const void *q, uint8_t *label_out, int32_t *nh_out, int D, int dtype,
                            int max_len, cudaStream_t s);
// shared memory of the identification kernels (single query, or multi:
// the ring's newest min(P, ntok) queries) for dense segments of up to
// max_len tokens; at most what update_prepare enabled
size_t identify_smem_bytes(int max_len, int P, bool grid2d, bool multi);
// multi-query Step 2 over the ring's newest min(P, ntok) queries
cudaError_t launch_identify_multi(const CacheArgs &c, const MethodArgs &m, int layer_base,
                                  int nheads, uint8_t *label_out, int32_t *nh_out, int D,
                                  int dtype, int max_len, cudaStream_t s);
// group > 0: the aggregate-preserving budgets over groups of that many heads
cudaError_t launch_budgets(const uint8_t *label, int32_t *budget, int32_t *cap, int64_t *off,
                           int n, int C, int B_g, int w, int P, int group, cudaStream_t s);

}  // namespace hkv
