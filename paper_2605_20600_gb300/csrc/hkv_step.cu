// One decode step of one layer in a single launch: attention of every head's
// new query over the head's retained tokens and the step's new token (Eq. 1),
// fused with the append of that token to the cache (Sec. 3, KV Cache).
//
// The split-K layout is the one of the two-kernel design in hkv_attention.cu
// (the layer's heads rounded up to whole tiles and concatenated; gridDim.x
// equal contiguous ranges, one per CTA; a warp-specialised TMA pipeline with
// a producer warp, consumer warps and an epilogue warp), but the work that
// the finishing kernel did there happens inside this launch:
//
//  * tile order: a CTA streams the start of the head that continues into a
//    later range first, then the piece of the head that began in an earlier
//    range, then the heads wholly inside its range. The piece a CTA streams
//    first is never the one that CTA combines, so a head in two pieces
//    never waits for a piece that finishes last in its CTA (measured: 0.3
//    us per step less than the other order at rho = 1/8);
//  * merges: a split head is combined by its first middle CTA (whose whole
//    range lies inside the head), else by the CTA holding its last row. The
//    other pieces write their partial result to the workspace as 64-bit
//    (value, launch epoch) pairs, which are single-copy atomic, so no fence
//    or flag is needed: the combining CTA's merge warp reads the pieces until
//    every pair carries this launch's epoch, while its consumers stream.
//    Pieces are combined in index order and the CTA's own piece last, so the
//    result does not depend on timing;
//  * prologue: every CTA reads the lengths of all the layer's heads to place
//    the ranges, but checks the other counters only for the heads of its own
//    range, in the same round of loads;
//  * appends and counters: every CTA arrives on a per-layer barrier word
//    once it is done reading the layer's counters (a CTA that found a bad
//    head marks its arrival); once the whole grid has arrived, and unless
//    one was marked, the merge warp copies the new token of every head
//    whose last row is in the CTA's range into the cache (nothing in the
//    launch reads those rows) and advances len, ntok and nbuf of those
//    heads, while the consumers stream. The next launch of the same layer
//    starts after this one completes, so the barrier word is free again by
//    then;
//  * programmatic dependent launch: with the prefetch flag the prologue and
//    the first tiles of old K/V rows go ahead of the wait for the previous
//    kernel; the step's inputs (q, the new k and v) are read after it;
//  * every wait is bounded (HKV_ERR_TIMEOUT in the error word).
//
// The lengths of every head whose range a CTA touches are kept in a table in
// shared memory (kStepTable heads); the host takes this path only when no
// range can hold more heads than that.
#include <math.h>
#include <stdlib.h>

#include "hkv_attn_common.cuh"
#include "hkv_device.cuh"
#include "hkv_kernels.h"

namespace hkv {
namespace {

#ifdef HKV_ATTN_TRACE
__device__ unsigned long long *g_step_trace = nullptr;  // [layer][kAttnMaxGrid][32]
#define STEP_TRACE_AT(slot) \
  g_step_trace[((size_t)(p.layer_base / p.nheads) * kAttnMaxGrid + blockIdx.x) * 32 + (slot)]
#define STEP_TRACE(slot)                                    \
  do {                                                      \
    if (g_step_trace) STEP_TRACE_AT(slot) = globaltimer(); \
  } while (0)
#define STEP_TRACE_SET(slot, v)                 \
  do {                                          \
    if (g_step_trace) STEP_TRACE_AT(slot) = (v); \
  } while (0)
#define STEP_CLK() clock64()
#else
#define STEP_CLK() 0ll
#define STEP_TRACE(slot) \
  do {                   \
  } while (0)
#define STEP_TRACE_SET(slot, v) \
  do {                          \
    (void)(v);                  \
  } while (0)
#endif

// Tuning knobs (compile time) of the one-launch step, per head dimension:
// consumer warps, bytes of K per stage, stages, tiles loaded before the wait,
// and the CTAs per SM the kernel is built to be resident with (the grid uses
// kStepActivePerSm). Measured per layer step (A/B in one process): rows of
// 256 B stream best with 8 consumer warps over 48-row tiles in 3 stages, all
// loaded before the wait (Lumina-mGPT 1024 at rho = 1/8: 13.01 us with 7
// warps over 42 rows and 2 before the wait, 12.77 with 8 over 48, 12.63
// with all 3 before it; 56-row tiles 13.06, 64-row tiles in 2 stages 13.10);
// rows of 128 B (LlamaGen-XL's short heads, many to a CTA) with 128-row
// tiles in 2 stages (15.26 us against 16.06 with 64-row tiles in 3 stages
// and 17.42 with 96-row tiles in 3).
#ifndef HKV_STEP_CW_D128
#define HKV_STEP_CW_D128 8
#endif
#ifndef HKV_STEP_TILE_BYTES_D128
#define HKV_STEP_TILE_BYTES_D128 12288
#endif
#ifndef HKV_STEP_STAGES_D128
#define HKV_STEP_STAGES_D128 3
#endif
#ifndef HKV_STEP_PRE_D128
#define HKV_STEP_PRE_D128 3
#endif
#ifndef HKV_STEP_CW_D64
#define HKV_STEP_CW_D64 8
#endif
#ifndef HKV_STEP_TILE_BYTES_D64
#define HKV_STEP_TILE_BYTES_D64 16384
#endif
#ifndef HKV_STEP_STAGES_D64
#define HKV_STEP_STAGES_D64 2
#endif
#ifndef HKV_STEP_PRE_D64
#define HKV_STEP_PRE_D64 1
#endif
#ifndef HKV_STEP_RESIDENT_PER_SM
#define HKV_STEP_RESIDENT_PER_SM 2
#endif

template <int D, typename T>
using StepShape =
    TileShape<D, T, D == 64 ? HKV_STEP_CW_D64 : HKV_STEP_CW_D128,
              D == 64 ? HKV_STEP_TILE_BYTES_D64 : HKV_STEP_TILE_BYTES_D128,
              D == 64 ? HKV_STEP_STAGES_D64 : HKV_STEP_STAGES_D128,
              D == 64 ? HKV_STEP_PRE_D64 : HKV_STEP_PRE_D128>;

struct StepTable {
  int h0, n;                      // heads h0 .. h0 + n - 1
  long long start[kStepTable];    // first index (slot space) of head h0 + j
  long long off[kStepTable];      // arena offset
  int vlen[kStepTable];           // len + 1 (the new token)
  int nbuf[kStepTable];
  int ntok[kStepTable];           // written by the append (epilogue warp)
  unsigned char label[kStepTable];
};

constexpr int kFirst = 1, kLast = 2, kDone = 4;

struct TileMeta {  // producer -> consumers, one per stage
  int h, n, flags;
  long long hs, he;  // the head's rows in the index space
};

struct SegMeta {  // consumers -> epilogue; h < 0: no more segments
  int h;
  long long hs, he;
};

// Tiles of a slot-aligned sub-range [g, b) of the index space, head by head,
// over the table (j: table index of the current head).
template <int TT>
struct StepIter {
  int j, hl;
  long long hs, g, b;
  __device__ __forceinline__ bool done() const { return g >= b; }
  __device__ __forceinline__ long long tile_end() const {
    long long e = g + TT;
    if (e > hs + hl) e = hs + hl;
    if (e > b) e = b;
    return e;
  }
  __device__ __forceinline__ void advance(const StepTable &t) {
    g += TT;
    if (g >= b) return;
    while (g >= hs + slot_len<TT>(hl) && j + 1 < t.n) {
      ++j;
      hs = t.start[j];
      hl = t.vlen[j];
    }
  }
};

// The split of a layer's index space [0, total) into the CTAs' ranges: CTA k
// streams [start(k), start(k + 1)), `chunk` slots each (whole tiles, at
// least two), the last ones possibly shorter or empty.
template <int TT>
struct Ranges {
  long long total, chunk;
  int G;
  // the range size (a 64-bit division: one thread computes it)
  __device__ static long long chunk_of(long long total, int G, long long min_chunk) {
    const long long c = slot_len<TT>((total + G - 1) / G);
    return c < min_chunk ? min_chunk : c;
  }
  __device__ long long start(int k) const {
    const long long s = (long long)k * chunk;
    return k >= G || s > total ? total : s;
  }
  __device__ int owner(long long slot) const { return (int)(slot / chunk); }  // CTA holding slot
};

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t *p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release(uint32_t *p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// A float and the epoch of the launch that wrote it, as one 64-bit word:
// single-copy atomic, so a reader that sees the epoch sees the value.
__device__ __forceinline__ void st_pair(unsigned long long *p, float v, uint32_t ep) {
  const unsigned long long w = ((unsigned long long)ep << 32) | __float_as_uint(v);
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(w) : "memory");
}
__device__ __forceinline__ bool ld_pair(const unsigned long long *p, uint32_t ep, float &v) {
  unsigned long long w;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(w) : "l"(p) : "memory");
  v = __uint_as_float((uint32_t)w);
  return (uint32_t)(w >> 32) == ep;
}

// Combines a split head's own piece (m1, l1, A1) with its other pieces,
// already combined (m2, l2, A2), and stores the output row: the same
// instructions wherever it runs, so the result does not depend on which
// warp does it.
template <int CPL>
__device__ __forceinline__ void combine_store(float m1, float l1, const float *A1, float m2,
                                              float l2, const float *A2, float *out) {
  const float mx = fmaxf(m1, m2);
  const float w1 = m1 == -INFINITY ? 0.f : exp2f(m1 - mx);
  const float w2 = m2 == -INFINITY ? 0.f : exp2f(m2 - mx);
  const float Lt = l1 * w1 + l2 * w2;
  float A[CPL];
#pragma unroll
  for (int c = 0; c < CPL; ++c) A[c] = fmaf(A1[c], w1, A2[c] * w2) / Lt;
  Vec<CPL>::st(out, A);
}

// threads: a producer warp, the consumer warps, the epilogue warp and the
// merge warp
template <int D, typename T>
__host__ __device__ constexpr int step_threads() {
  return StepShape<D, T>::kThreads + 32;
}

template <int D, typename T>
__global__ void __launch_bounds__(step_threads<D, T>(), HKV_STEP_RESIDENT_PER_SM)
    step_kernel(const AttnArgs p) {
  using S = StepShape<D, T>;
  constexpr int kCW = S::kCW, kThr = step_threads<D, T>();
  constexpr int LPR = S::kLPR, EPL = S::kEPL, RPW = S::kRPW, TT = S::kTT;
  constexpr int RB = S::kRB, NS = S::kNS;
  constexpr int NST = kCW * RPW;  // row-group states per segment
  constexpr int CPL = D / 32;     // output channels per epilogue lane
  static_assert(NST <= 32, "a lane of the epilogue per state");
  static_assert(kStepTable <= kThr, "a thread per table entry");
  using V = Vec<CPL>;

  extern __shared__ __align__(128) unsigned char stages[];
  __shared__ uint64_t full[NS], empty[NS];
  __shared__ uint64_t epi_full[2], epi_free[2];  // two hand-over buffers
  __shared__ __align__(16) float red_acc[2][NST][D];
  __shared__ float red_m[2][NST], red_l[2][NST];
  __shared__ TileMeta meta[NS];
  __shared__ SegMeta seg[2];
  __shared__ StepTable tab;
  __shared__ long long scan_scratch[33];
  __shared__ long long s_s0, s_mg_k0, s_a, s_b, s_chunk;
  __shared__ int s_h0, s_h1, s_bad;
  __shared__ int s_mg_h, s_mg_j, s_mg_np;  // the split head this CTA combines
  __shared__ uint32_t s_ep;                // the launch's epoch
  // hand-overs between the epilogue and the merge warp: the epoch and the
  // merge head (ep_bar), the other pieces combined (oth_bar), and this CTA's
  // own piece or the news that the epilogue combined it already (own_bar)
  __shared__ uint64_t ep_bar, oth_bar, own_bar;
  __shared__ __align__(16) float own_acc[D], oth_acc[D];
  __shared__ float own_ml[2], oth_ml[2];
  __shared__ int s_own_state;  // 1: combined by the epilogue, 2: own piece handed over
  __shared__ volatile int s_abort;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nheads = p.nheads;
  const int G = gridDim.x;
  const int bx = blockIdx.x;

  if (tid == 0) {
    STEP_TRACE(0);
#ifdef HKV_ATTN_TRACE
    if (g_step_trace) {
      unsigned smid;
      asm volatile("mov.u32 %0, %%smid;" : "=r"(smid));
      STEP_TRACE_AT(16) = smid;
    }
#endif
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kCW);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&epi_full[s], kCW);
      mbar_init(&epi_free[s], 1);
    }
    mbar_init(&ep_bar, 32);
    mbar_init(&oth_bar, 32);
    mbar_init(&own_bar, 32);
    fence_barrier_init();
    s_abort = 0;
    s_bad = 0;
    s_h0 = 0;
    s_h1 = -1;
    s_s0 = 0;
    s_mg_h = -1;
  }
  if (!p.prefetch) pdl_wait();

  // ---- prologue: the layer's lengths, one round of loads -------------------
  // Every thread takes a contiguous slice of the layer's heads and sums
  // their slots; a block scan gives each slice its first index, so every
  // CTA computes the same ranges, and a negative length stops every CTA.
  // Offsets, capacities, labels and buffer counts are checked only for the
  // heads of the CTA's own range: a CTA that finds a bad one streams nothing
  // and flags the step on the layer's barrier word, and no CTA then appends
  // or advances a counter. All of it takes one round of loads: a slice of
  // one head is read whole into registers; with longer slices only the
  // lengths are, and the same round reads the other counters of a window of
  // kThr heads around the range's expected place (heads of equal length). A
  // range outside the window reads them once it is known.
  const int per = (nheads + kThr - 1) / kThr;
  const int h_lo = tid * per < nheads ? tid * per : nheads;
  const int h_hi = h_lo + per < nheads ? h_lo + per : nheads;
  const bool in_regs = per <= 1;
  long long mine = 0;
  int bad = 0;
  auto count = [&](int l) {
    if (l < 0) bad = HKV_ERR_BOUNDS;
    mine += slot_len<TT>(l + 1);
  };
  // the counters of one head in registers: this thread's slice (in_regs) or
  // its head of the window
  int rl = 0, rcp = 0, rnb = 0, rlb = 0;
  long long ro = 0;
  int win_lo = 0;
  if (in_regs) {
    if (h_lo < h_hi) {  // every load issued before any use
      rl = p.len[h_lo];
      ro = p.off[h_lo];
      rcp = p.cap[h_lo];
      rlb = p.label[p.layer_base + h_lo];
      rnb = p.nbuf[p.layer_base + h_lo];
      count(rl);
    }
  } else {
    const int guess = (int)((float)bx * ((float)nheads / (float)G));
    win_lo = guess - kThr / 2;
    win_lo = win_lo < nheads - kThr ? win_lo : nheads - kThr;
    win_lo = win_lo > 0 ? win_lo : 0;
    const int wh = win_lo + tid;
    if (wh < nheads) {
      ro = p.off[wh];
      rcp = p.cap[wh];
      rlb = p.label[p.layer_base + wh];
      rnb = p.nbuf[p.layer_base + wh];
    }
#pragma unroll 4
    for (int h = h_lo; h < h_hi; ++h) count(p.len[h]);
  }
  long long total;
  const long long slice_start = block_excl_scan<long long>(mine, scan_scratch, &total);
  if (tid == 0) STEP_TRACE(10);
  if (bad) s_bad = bad;
  if (tid == 0) {  // this CTA's range (a 64-bit division: one thread)
    Ranges<TT> r0;
    r0.total = total;
    r0.G = G;
    r0.chunk = Ranges<TT>::chunk_of(total, G, S::kMinChunk);
    s_chunk = r0.chunk;
    s_a = r0.start(bx);
    s_b = r0.start(bx + 1);
  }
  __syncthreads();
  Ranges<TT> rg;
  rg.total = total;
  rg.G = G;
  rg.chunk = s_chunk;
  if (s_bad) {  // every CTA sees it: none reads further or arrives
    pdl_wait();
    if (bx == 0 && tid == 0) set_err(p.err, (uint32_t)s_bad);
    return;
  }
  const long long a = s_a, b = s_b;
  bool active = a < total;
  if (active && mine > 0) {  // the heads holding the range's first and last index
    const bool has_a = slice_start <= a && a < slice_start + mine;
    const bool has_b = slice_start <= b - 1 && b - 1 < slice_start + mine;
    if (has_a || has_b) {
      long long st = slice_start;
      auto visit = [&](int h, int l) {
        const long long L = slot_len<TT>(l + 1);
        if (has_a && a >= st && a < st + L) {
          s_h0 = h;
          s_s0 = st;
        }
        if (has_b && b - 1 >= st && b - 1 < st + L) s_h1 = h;
        st += L;
      };
      if (in_regs) {
        visit(h_lo, rl);
      } else {
        for (int h = h_lo; h < h_hi; ++h) visit(h, p.len[h]);
      }
    }
  }
  __syncthreads();
  if (tid == 0) STEP_TRACE(11);
  int n = active ? s_h1 - s_h0 + 1 : 0;
  int own_bad = 0;
  if (n > kStepTable) {  // excluded by the host; the step is not taken
    own_bad = HKV_ERR_CAPACITY;
    n = 0;
    active = false;
  }
  const int h0 = s_h0;
  // the table entry of head h with its checks
  auto enter = [&](int h, long long st, int l, long long o, int cp, int lab, int nb) {
    const int j = h - h0;
    int e = 0;
    if (o < 0 || o + cp > p.arena_tokens) e = HKV_ERR_BOUNDS;
    else if (l + 1 > cp) e = HKV_ERR_CAPACITY;
    else if (lab != HKV_DENSE && nb >= p.period) e = HKV_ERR_STATE;  // the update is due first
    if (e) atomicMax(&s_bad, e);
    if (st >= 0) {
      tab.start[j] = st;
      tab.vlen[j] = l + 1;
    }
    tab.off[j] = o;
    tab.nbuf[j] = nb;
    tab.label[j] = (unsigned char)lab;
  };
  if (in_regs) {  // the slice owner enters its head
    if (active && h_lo < h_hi && h_lo >= h0 && h_lo < h0 + n)
      enter(h_lo, slice_start, rl, ro, rcp, rlb, rnb);
  } else {
    // the slice owners place the range's heads in the index space ...
    if (active && h_lo <= h0 + n - 1 && h_hi > h0) {
      long long st = slice_start;
      for (int h = h_lo; h < h_hi && h < h0 + n; ++h) {
        const int l = p.len[h];
        if (h >= h0) {
          tab.start[h - h0] = st;
          tab.vlen[h - h0] = l + 1;
        }
        st += slot_len<TT>(l + 1);
      }
    }
    // ... and a thread per head checks the rest: from registers when the
    // window holds the whole range, else from one more round of loads
    const bool in_win = h0 >= win_lo && h0 + n <= win_lo + kThr;
    const int jt = in_win ? win_lo + tid - h0 : tid;
    if (active && jt >= 0 && jt < n) {
      const int h = h0 + jt, i = p.layer_base + h;
      if (in_win)
        enter(h, -1, p.len[h], ro, rcp, rlb, rnb);
      else
        enter(h, -1, p.len[h], p.off[h], p.cap[h], p.label[i], p.nbuf[i]);
    }
  }
  if (tid == 0) {
    tab.h0 = h0;
    tab.n = n;
  }
  __syncthreads();
  if (s_bad) {  // a bad head in this range: stream nothing
    own_bad = own_bad > s_bad ? own_bad : s_bad;
    active = false;
  }
  // From here on nothing reads the layer's counters in global memory: the
  // merge warp arrives on the layer's barrier word below.
  if (tid == 0) STEP_TRACE(1);

  // ---- the range's sub-ranges, in streaming order --------------------------
  // S: the piece of the head that began before a; E: the start of the head
  // that continues past b; M: the heads in between.
  long long sub_g[3], sub_b[3];
  int sub_j[3], nsub = 0;
  if (active) {
    const long long hs0 = tab.start[0];
    const long long se0 = hs0 + slot_len<TT>(tab.vlen[0]);
    const long long hs1 = tab.start[n - 1];
    const long long he1 = hs1 + tab.vlen[n - 1];
    const bool has_s = hs0 < a;
    const bool has_e = he1 > b && (n > 1 || !has_s);
    const long long s_end = se0 < b ? se0 : b;
    const long long e_beg = hs1 > a ? hs1 : a;
    if (has_e) {
      sub_g[nsub] = e_beg, sub_b[nsub] = b, sub_j[nsub] = n - 1;
      ++nsub;
    }
    if (has_s) {
      sub_g[nsub] = a, sub_b[nsub] = s_end, sub_j[nsub] = 0;
      ++nsub;
    }
    const long long m_lo = has_s ? s_end : a, m_hi = has_e ? e_beg : b;
    if (m_lo < m_hi) {
      sub_g[nsub] = m_lo, sub_b[nsub] = m_hi, sub_j[nsub] = has_s ? 1 : 0;
      ++nsub;
    }
  }

  if (tid == 0) STEP_TRACE(12);

  // ---- producer state (warp 0, lane 0) ------------------------------------
  const bool producer = tid == 0;
  StepIter<TT> pit;
  int sr = 0;  // current sub-range
  auto start_sub = [&](int r) {
    pit.j = sub_j[r];
    pit.hs = tab.start[pit.j];
    pit.hl = tab.vlen[pit.j];
    pit.g = sub_g[r];
    pit.b = sub_b[r];
  };
  pit.g = pit.b = 0;
  pit.j = 0;
  pit.hs = 0;
  pit.hl = 0;
  if (nsub > 0) start_sub(0);
  auto more = [&]() {  // moves to the next sub-range when one is exhausted
    while (pit.done() && sr + 1 < nsub) start_sub(++sr);
    return !pit.done();
  };
  int issued = 0;
  // the arena rows are read once per step: evict them from L2 first (measured:
  // 0.4-0.55 us per step slower without the hint)
  const uint64_t stream_pol = producer ? l2_evict_first_policy() : 0;
  struct Pending {
    int h, slot_new;
    bool first, has_new;
  };
  auto issue_old = [&](Pending &pd) {  // describe, expect and copy the arena rows
    const int stage = issued % NS;
    const long long ge = pit.tile_end();
    const long long he = pit.hs + pit.hl;
    const int r0 = (int)(pit.g - pit.hs), r1 = (int)(ge - pit.hs);
    const int real = pit.hl - 1;  // rows in the arena
    const int n_old = (r1 < real ? r1 : real) - r0;
    unsigned char *dk = stages + stage * S::kStageBytes;
    const int h = h0 + pit.j;
    pd.h = h;
    pd.slot_new = real - r0;
    pd.first = pit.g == pit.hs || pit.g == sub_g[sr];
    pd.has_new = r1 == pit.hl;
    TileMeta &mt = meta[stage];
    mt.h = h;
    mt.n = (int)(ge - pit.g);
    mt.flags = (pd.first ? kFirst : 0) | (ge == (pit.b < he ? pit.b : he) ? kLast : 0);
    mt.hs = pit.hs;
    mt.he = he;
    if (n_old > 0) {
      const uint32_t bytes = (uint32_t)n_old * RB;
      const long long row = tab.off[pit.j] + r0;
      mbar_expect_tx(&full[stage], 2 * bytes);
      bulk_g2s_hint(dk, static_cast<const unsigned char *>(p.K) + row * RB, bytes, &full[stage],
                    stream_pol);
      bulk_g2s_hint(dk + TT * RB, static_cast<const unsigned char *>(p.V) + row * RB, bytes,
                    &full[stage], stream_pol);
    }
    pit.advance(tab);
    ++issued;
  };
  auto issue_extra = [&](const Pending &pd, int stage) {  // the step's inputs, then arrive
    unsigned char *dk = stages + stage * S::kStageBytes;
    unsigned char *dv = dk + TT * RB;
    mbar_arrive_expect_tx(&full[stage], (pd.has_new ? 2 * RB : 0) + (pd.first ? RB : 0));
    if (pd.has_new) {
      bulk_g2s(dk + pd.slot_new * RB,
               static_cast<const unsigned char *>(p.k_new) + (size_t)pd.h * RB, RB, &full[stage]);
      bulk_g2s(dv + pd.slot_new * RB,
               static_cast<const unsigned char *>(p.v_new) + (size_t)pd.h * RB, RB, &full[stage]);
    }
    if (pd.first)
      bulk_g2s(dv + TT * RB, static_cast<const unsigned char *>(p.q) + (size_t)pd.h * RB, RB,
               &full[stage]);
  };
  Pending pre[NS];
  int n_pre = 0;
  if (producer)
    for (; n_pre < (p.prefetch ? S::kPre : NS) && more(); ++n_pre) issue_old(pre[n_pre]);
  if (tid == 0) STEP_TRACE(7);

  if (p.prefetch) pdl_wait();  // the step's inputs are visible from here on
  if (tid == 0) STEP_TRACE(2);
  pdl_launch_dependents();

  if (warp == 0) {
    // ---- producer ----------------------------------------------------------
    if (producer) {
      long long w_empty = 0;  // cycles waiting for free stages (tracer)
      int armed = 0;  // stages whose producer arrival is done (issued order)
#pragma unroll
      for (int j = 0; j < NS; ++j)
        if (j < n_pre) issue_extra(pre[j], j);
      armed = n_pre;
      while (more()) {
        const int stage = issued % NS;
        const long long c0 = STEP_CLK();
        if (s_abort ||
            (issued >= NS && !mbar_wait(&empty[stage], (uint32_t)(issued / NS - 1) & 1u))) {
          s_abort = 1;
          set_err(p.err, HKV_ERR_TIMEOUT);
          break;
        }
        w_empty += STEP_CLK() - c0;
        Pending pd;
        issue_old(pd);
        issue_extra(pd, stage);
        armed = issued;
      }
      if (!s_abort) {  // no more tiles: a closing record for the consumers
        const int stage = issued % NS;
        if (issued >= NS && !mbar_wait(&empty[stage], (uint32_t)(issued / NS - 1) & 1u)) {
          s_abort = 1;
          set_err(p.err, HKV_ERR_TIMEOUT);
        } else {
          meta[stage].flags = kDone;
          mbar_arrive(&full[stage]);
        }
      }
      STEP_TRACE_SET(20, w_empty);
      if (s_abort) {
        // No bulk copy may land in shared memory after the CTA exits: wait
        // (bounded) for every armed stage that may still be in flight. A
        // stage reused after an empty-barrier wait is complete already.
        const int first = armed - NS > 0 ? armed - NS : 0;
        for (int t = first; t < armed; ++t) mbar_wait(&full[t % NS], (uint32_t)(t / NS) & 1u);
      }
    }
  } else if (warp <= kCW) {
    // ---- consumers ---------------------------------------------------------
    const int ctid = tid - 32, cw = warp - 1;
    const int grp = lane / LPR, col = lane % LPR;
    using M = LaneMath<T>;
    static_assert(M::kEPL == EPL, "lane mapping");
    typename M::Q q;
    float2 acc[EPL / 2];
    float m = -INFINITY, l = 0.f;
    int nseg = 0;
#pragma unroll
    for (int e = 0; e < EPL / 2; ++e) acc[e] = make_float2(0.f, 0.f);
    int n_tiles = 0;
    long long w_full = 0, w_hand = 0;  // cycles waiting for tiles, for the epilogue (tracer)
    // hands one segment's state (or the closing record) to the epilogue
    auto hand_over = [&](const SegMeta *sm) {
      const int bb = nseg & 1;
      const long long c0 = STEP_CLK();
      if (nseg >= 2 && !s_abort &&
          !mbar_wait(&epi_free[bb], (uint32_t)((nseg >> 1) - 1) & 1u)) {
        s_abort = 1;
        set_err(p.err, HKV_ERR_TIMEOUT);
      }
      w_hand += STEP_CLK() - c0;
      if (sm) {
        const int si = cw * RPW + grp;
        float2 *dst = reinterpret_cast<float2 *>(&red_acc[bb][si][col * EPL]);
#pragma unroll
        for (int e = 0; e < EPL / 2; ++e) dst[e] = acc[e];
        if (col == 0) {
          red_m[bb][si] = m;
          red_l[bb][si] = l;
        }
        if (cw == 0 && lane == 0) seg[bb] = *sm;
      } else if (cw == 0 && lane == 0) {
        seg[bb].h = -1;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&epi_full[bb]);
      ++nseg;
    };
    for (int tile = 0;; ++tile) {
      const int stage = tile % NS;
      const long long c0 = STEP_CLK();
      if (!s_abort && !mbar_wait(&full[stage], (uint32_t)(tile / NS) & 1u)) {
        s_abort = 1;
        set_err(p.err, HKV_ERR_TIMEOUT);
      }
      if (tile > 0) w_full += STEP_CLK() - c0;
      if (s_abort) break;
      const int flags = meta[stage].flags;
      if (flags & kDone) break;
      if (tile == 0 && ctid == 0) STEP_TRACE(3);
      ++n_tiles;
      const int nr = meta[stage].n;
      const unsigned char *Ks = stages + stage * S::kStageBytes;
      const unsigned char *Vs = Ks + TT * RB;
      if (flags & kFirst) {  // first tile of this head in this piece
        M::load_q(q, *reinterpret_cast<const uint4 *>(Vs + TT * RB + col * 16), p.qscale);
#pragma unroll
        for (int e = 0; e < EPL / 2; ++e) acc[e] = make_float2(0.f, 0.f);
        m = -INFINITY;
        l = 0.f;
      }
      float sc[S::kSteps];
#pragma unroll
      for (int st = 0; st < S::kSteps; ++st) {
        const int r = st * (kCW * RPW) + cw * RPW + grp;
        float dot = 0.f;
        if (r < nr) dot = M::dot(q, *reinterpret_cast<const uint4 *>(Ks + r * RB + col * 16));
#pragma unroll
        for (int o = LPR / 2; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xFFFFFFFFu, dot, o);
        sc[st] = r < nr ? M::score(dot, p.qscale) : -INFINITY;
      }
      float mt = sc[0];
#pragma unroll
      for (int st = 1; st < S::kSteps; ++st) mt = fmaxf(mt, sc[st]);
      const float mn = fmaxf(m, mt);
      if (mn != -INFINITY) {
        const float corr = ex2_approx(m - mn);  // measured: 0.11 us per step less than exp2f
        l *= corr;
#pragma unroll
        for (int e = 0; e < EPL / 2; ++e) acc[e] = __fmul2_rn(acc[e], make_float2(corr, corr));
#pragma unroll
        for (int st = 0; st < S::kSteps; ++st) {
          const int r = st * (kCW * RPW) + cw * RPW + grp;
          if (r < nr) {
            const float pr = ex2_approx(sc[st] - mn);
            l += pr;
            M::add_v(acc, *reinterpret_cast<const uint4 *>(Vs + r * RB + col * 16), pr);
          }
        }
        m = mn;
      }
      if (flags & kLast) {  // last tile of this head in this piece: hand it over
        SegMeta sm;
        sm.h = meta[stage].h;
        sm.hs = meta[stage].hs;
        sm.he = meta[stage].he;
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[stage]);
        hand_over(&sm);
      } else {
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[stage]);
      }
    }
    if (ctid == 0) STEP_TRACE(4);
    if (ctid == 0) STEP_TRACE_SET(17, n_tiles);
    hand_over(nullptr);  // nothing more
    if (ctid == 0) STEP_TRACE_SET(21, w_full);
    if (ctid == 0) STEP_TRACE_SET(22, w_hand);
  } else if (warp == kCW + 1) {
    // ---- epilogue: combine each segment's row-group states ----------------
    bool have_ep = false;  // the epoch and the merge head (merge warp)
    long long w_epi = 0;   // cycles waiting for segments (tracer)
    int k = 0;
    for (;; ++k) {
      const int bb = k & 1;
      const long long c0 = STEP_CLK();
      if (!s_abort && !mbar_wait(&epi_full[bb], (uint32_t)(k >> 1) & 1u)) {
        s_abort = 1;
        set_err(p.err, HKV_ERR_TIMEOUT);
      }
      if (k > 0) w_epi += STEP_CLK() - c0;
      if (s_abort) break;
      const SegMeta sg = seg[bb];
      if (sg.h < 0) break;
      const int h = sg.h;
      const long long hs = sg.hs, he = sg.he;
      // lane s < NST weighs state s
      const float ms = lane < NST ? red_m[bb][lane] : -INFINITY;
      float mx = ms;
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
      const float ws = ms == -INFINITY ? 0.f : exp2f(ms - mx);
      float L = lane < NST ? red_l[bb][lane] * ws : 0.f;
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) L += __shfl_xor_sync(0xFFFFFFFFu, L, o);
      float A[CPL];
#pragma unroll
      for (int c = 0; c < CPL; ++c) A[c] = 0.f;
#pragma unroll
      for (int si = 0; si < NST; ++si) {
        const float sw = __shfl_sync(0xFFFFFFFFu, ws, si);
        float r[CPL];
        V::lds(&red_acc[bb][si][CPL * lane], r);
#pragma unroll
        for (int c = 0; c < CPL; ++c) A[c] = fmaf(r[c], sw, A[c]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&epi_free[bb]);  // the consumers may reuse the buffer
      const bool whole = hs >= a && he <= b;
      if (!whole && !have_ep) {
        if (!mbar_wait(&ep_bar, 0u)) {
          s_abort = 1;
          set_err(p.err, HKV_ERR_TIMEOUT);
          break;
        }
        have_ep = true;
      }
      if (whole) {  // the whole head is in this CTA's range
#pragma unroll
        for (int c = 0; c < CPL; ++c) A[c] /= L;
        V::st(p.out + (size_t)h * D + CPL * lane, A);
      } else if (h == s_mg_h) {  // this CTA combines the head
        // the other pieces already combined by the merge warp: finish here;
        // else hand this piece to the merge warp
        int ready = mbar_test_wait(&oth_bar, 0u) ? 1 : 0;
        ready = __shfl_sync(0xFFFFFFFFu, ready, 0);
        if (ready) {
          mbar_wait(&oth_bar, 0u);  // complete: every lane acquires oth_*
          float A2[CPL];
          V::lds(&oth_acc[CPL * lane], A2);
          combine_store<CPL>(mx, L, A, oth_ml[0], oth_ml[1], A2,
                             p.out + (size_t)h * D + CPL * lane);
          STEP_TRACE_SET(18, globaltimer());
        } else {
          V::st(&own_acc[CPL * lane], A);
          if (lane == 0) {
            own_ml[0] = mx;
            own_ml[1] = L;
          }
        }
        if (lane == 0) s_own_state = ready ? 1 : 2;
        __syncwarp();
        mbar_arrive(&own_bar);  // all 32 lanes
      } else {  // a piece for the combining CTA: epoch-tagged, no fence needed
        unsigned long long *ps = p.pslot + ((size_t)bx * 2 + (hs < a ? 1 : 0)) * (D + 2);
#pragma unroll
        for (int c = 0; c < CPL; ++c) st_pair(ps + CPL * lane + c, A[c], s_ep);
        if (lane == 0) {
          st_pair(ps + D, mx, s_ep);
          st_pair(ps + D + 1, L, s_ep);
        }
      }
    }
    if (lane == 0) STEP_TRACE(5);
    STEP_TRACE_SET(9, k);
    if (lane == 0) STEP_TRACE_SET(23, w_epi);
  } else {
    // ---- merge warp: barrier, appends, counters, the combined split head ---
    // The split head this CTA combines, if any: the head of its range's
    // first index when this CTA is that head's first middle CTA (its whole
    // range inside the head) or, for a head in two pieces, holds its last
    // row. Then the launch's epoch, unique per (layer, launch of that
    // layer), from the generation of the layer's barrier word; the epilogue
    // waits for both only when it meets a split head.
    constexpr uint32_t kBadStep = 0x80000000u;  // in the generation: step not taken
    uint32_t gen0 = 0;
    if (lane == 0) {
      if (active && tab.start[0] < a) {
        const long long hs0 = tab.start[0], he0 = hs0 + tab.vlen[0];
        const long long k0 = rg.owner(hs0), k1 = rg.owner(he0 - 1);
        const long long np = k1 - k0 + 1;
        if ((np >= 3 ? k0 + 1 : k1) == bx) {
          s_mg_k0 = k0;
          s_mg_np = (int)np;
          s_mg_j = (int)(bx - k0);
          s_mg_h = h0;
        }
      }
      gen0 = ld_acquire(p.bar + 1);
      s_ep = ((gen0 & ~kBadStep) + 1u) * (uint32_t)p.n_layers + (uint32_t)(p.layer_base / nheads);
    }
    __syncwarp();
    mbar_arrive(&ep_bar);  // all 32 lanes: the epilogue may read s_ep, s_mg_*
    // Arrive on the layer's barrier words {arrivals, generation, worst
    // status}: this CTA is done reading counters. The last of the grid to
    // arrive resets the count and publishes the next generation, which the
    // others watch. A CTA with a bad head raises the worst status and adds
    // 1 << 16 more; the last arriver then marks the generation (the step is
    // not taken) and reports the worst status, the same whichever CTAs found
    // bad heads first.
    const uint32_t inc = own_bad ? 0x10001u : 1u;
    uint32_t gen1 = 0;
    int bar_done = 0;
    if (lane == 0) {
      if (own_bad) {
        atomicMax(p.bar + 2, (uint32_t)own_bad);
        __threadfence();  // the status before the arrival
      }
      const uint32_t old = atomicAdd(p.bar, inc);
      if ((old & 0xFFFFu) == (uint32_t)G - 1) {
        const bool bad_step = ((old + inc) >> 16) != 0;
        if (bad_step) {
          __threadfence();  // the bad CTAs' statuses after their arrivals
          set_err(p.err, atomicExch(p.bar + 2, 0u));
        }
        p.bar[0] = 0;
        gen1 = (((gen0 & ~kBadStep) + 1u) & ~kBadStep) | (bad_step ? kBadStep : 0u);
        st_release(p.bar + 1, gen1);
        bar_done = 1;
      }
    }
    gen0 = __shfl_sync(0xFFFFFFFFu, gen0, 0);
    bar_done = __shfl_sync(0xFFFFFFFFu, bar_done, 0);
    const uint64_t t0 = globaltimer();
    auto timed_out = [&]() {
      if (globaltimer() - t0 <= kWaitTimeoutNs) return false;
      if (lane == 0) {
        s_abort = 1;
        set_err(p.err, HKV_ERR_TIMEOUT);
      }
      return true;
    };
    if (own_bad) {
      // empty pieces in both of this CTA's slots, so that no combining CTA
      // waits for them (the step is not taken; the outputs are not defined)
      for (int sl = 0; sl < 2; ++sl) {
        unsigned long long *ps = p.pslot + ((size_t)bx * 2 + sl) * (D + 2);
        for (int c = lane; c < D; c += 32) st_pair(ps + c, 0.f, s_ep);
        if (lane == 0) {
          st_pair(ps + D, -INFINITY, s_ep);
          st_pair(ps + D + 1, 0.f, s_ep);
        }
      }
    }

    while (!s_abort && !bar_done) {
      if (lane == 0) {
        gen1 = ld_acquire(p.bar + 1);
        bar_done = gen1 != gen0;
      }
      bar_done = __shfl_sync(0xFFFFFFFFu, bar_done, 0);
      if (!bar_done && timed_out()) break;
    }
    gen1 = __shfl_sync(0xFFFFFFFFu, gen1, 0);
    __syncwarp();
    STEP_TRACE_SET(19, globaltimer());
    const bool taken = !s_abort && bar_done && !(gen1 & kBadStep) && active;

    // Appends: the CTA holding a head's last row writes the new token (K/V
    // row at index len, its position, q into the ring of the periodic
    // update), then advances that head's counters. Nothing in this launch
    // reads them; they wait for the barrier only to learn whether the step
    // is taken, which it is by then long before the consumers finish.
    if (taken) {
      for (int j0 = 0; j0 < n; j0 += 32) {  // ntok of 32 heads per round
        const int j = j0 + lane;
        if (j < n && tab.start[j] + tab.vlen[j] > a && tab.start[j] + tab.vlen[j] <= b)
          tab.ntok[j] = p.ntok[p.layer_base + h0 + j];
      }
      __syncwarp();
      // the K, V and q rows of every appended head as 16-byte chunks, a
      // lane per chunk, every load of a round issued before its stores
      constexpr int CH = RB / 16;  // chunks of a row
      constexpr int NU = 8;        // chunks per lane and round
      // The appended heads (a < he <= b) are the table's first napp entries:
      // the first head's rows always reach past a, and only the last head
      // can continue past b.
      const int napp = tab.start[n - 1] + tab.vlen[n - 1] <= b ? n : n - 1;
      constexpr int first_app = 0;
      const int units = napp * 3 * CH;
      for (int u0 = 0; u0 < units; u0 += 32 * NU) {
        uint4 x[NU];
        unsigned char *dst[NU];
#pragma unroll
        for (int v = 0; v < NU; ++v) {
          const int u = u0 + v * 32 + lane;
          dst[v] = nullptr;
          if (u < units) {
            const int jj = first_app + u / (3 * CH), w3 = (u / CH) % 3, cc = u % CH;
            const int h = h0 + jj, i = p.layer_base + h;
            const unsigned char *src = w3 == 0 ? static_cast<const unsigned char *>(p.k_new)
                                     : w3 == 1 ? static_cast<const unsigned char *>(p.v_new)
                                               : static_cast<const unsigned char *>(p.q);
            x[v] = reinterpret_cast<const uint4 *>(src + (size_t)h * RB)[cc];
            const long long row = tab.off[jj] + tab.vlen[jj] - 1;
            unsigned char *d = w3 == 0 ? static_cast<unsigned char *>(p.K) + row * RB
                             : w3 == 1 ? static_cast<unsigned char *>(p.V) + row * RB
                                       : static_cast<unsigned char *>(p.qbuf) +
                                             ((size_t)i * p.period + tab.ntok[jj] % p.period) * RB;
            dst[v] = d + (size_t)cc * 16;
          }
        }
#pragma unroll
        for (int v = 0; v < NU; ++v)
          if (dst[v]) *reinterpret_cast<uint4 *>(dst[v]) = x[v];
      }
      for (int jj = first_app + lane; jj < first_app + napp; jj += 32)
        p.pos[tab.off[jj] + tab.vlen[jj] - 1] = p.n_cond + tab.ntok[jj];
    }
    STEP_TRACE_SET(8, globaltimer());
    if (taken) {
      for (int j = lane; j < n; j += 32) {
        const long long hs = tab.start[j], he = hs + tab.vlen[j];
        if (he > a && he <= b) {
          const int h = h0 + j, i = p.layer_base + h;
          p.len[h] = tab.vlen[j];
          p.ntok[i] = tab.ntok[j] + 1;
          if (tab.label[j] != HKV_DENSE) p.nbuf[i] = tab.nbuf[j] + 1;
        }
      }
    }

    // The split head this CTA combines: the other pieces, combined in index
    // order once all of them carry this launch's epoch, then this CTA's own
    // piece (from the epilogue), so the result does not depend on timing.
    const int mh = s_mg_h;
    if (mh >= 0 && !s_abort) {
      const int np = s_mg_np, mj = s_mg_j;
      const long long k0 = s_mg_k0;
#ifdef HKV_STEP_TEST_STALL
      // test builds only: wait for an epoch no launch writes, so that the
      // bounded wait runs out (HKV_ERR_TIMEOUT) with no bulk copy involved
      const uint32_t want = s_ep + 1u;
#else
      const uint32_t want = s_ep;
#endif
      float om = -INFINITY, ol = 0.f, oA[CPL];
#pragma unroll
      for (int c = 0; c < CPL; ++c) oA[c] = 0.f;
      for (;;) {
        bool ready = true;
        om = -INFINITY;
        ol = 0.f;
#pragma unroll
        for (int c = 0; c < CPL; ++c) oA[c] = 0.f;
        for (int t = 0; t < np && ready; ++t) {
          if (t == mj) continue;
          // piece t: the end piece of CTA k0, the start piece of the others
          const unsigned long long *ps = p.pslot + ((size_t)(k0 + t) * 2 + (t > 0 ? 1 : 0)) * (D + 2);
          float At[CPL], mt, lt;
          bool ok = true;
#pragma unroll
          for (int c = 0; c < CPL; ++c) ok &= ld_pair(ps + CPL * lane + c, want, At[c]);
          ok &= ld_pair(ps + D, want, mt);
          ok &= ld_pair(ps + D + 1, want, lt);
          ready = __all_sync(0xFFFFFFFFu, ok);
          if (!ready) break;
          const float mn = fmaxf(om, mt);
          const float co = om == -INFINITY ? 0.f : exp2f(om - mn);
          const float ct = mt == -INFINITY ? 0.f : exp2f(mt - mn);
          ol = ol * co + lt * ct;
#pragma unroll
          for (int c = 0; c < CPL; ++c) oA[c] = fmaf(At[c], ct, oA[c] * co);
          om = mn;
        }
        if (ready || timed_out()) break;
      }
      // hand the combined other pieces to the epilogue (not after a wait
      // that ran out: the head's output is then not written)
      if (!s_abort) {
        V::st(&oth_acc[CPL * lane], oA);
        if (lane == 0) {
          oth_ml[0] = om;
          oth_ml[1] = ol;
        }
        __syncwarp();
        mbar_arrive(&oth_bar);  // all 32 lanes
      }
      // this CTA's own piece, unless the epilogue combined it already
      while (!s_abort && !mbar_try_wait(&own_bar, 0u))
        if (timed_out()) break;
      __syncwarp();
      if (!s_abort && s_own_state == 2) {
        mbar_wait(&own_bar, 0u);  // complete: every lane acquires own_*
        float A1[CPL];
        V::lds(&own_acc[CPL * lane], A1);
        combine_store<CPL>(own_ml[0], own_ml[1], A1, om, ol, oA,
                           p.out + (size_t)mh * D + CPL * lane);
        STEP_TRACE_SET(18, globaltimer());
      }
    }
    if (lane == 0) STEP_TRACE(6);
  }
}

template <int D, typename T>
size_t step_smem() {
  return (size_t)StepShape<D, T>::kNS * StepShape<D, T>::kStageBytes;
}

template <int D, typename T>
cudaError_t step_prepare_t(int *ctas) {
  const size_t smem = step_smem<D, T>();
  cudaError_t e = cudaFuncSetAttribute(step_kernel<D, T>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas, step_kernel<D, T>,
                                                       step_threads<D, T>(), smem);
}

template <int D, typename T>
cudaError_t step_launch_t(const AttnArgs &a, int grid, cudaStream_t s) {
  static const bool pdl = getenv("HKV_NO_PDL") == nullptr;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(step_threads<D, T>());
  cfg.dynamicSmemBytes = step_smem<D, T>();
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  int na = 0;
  if (pdl) {
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
  }
  cfg.attrs = attr;
  cfg.numAttrs = na;
  return cudaLaunchKernelEx(&cfg, step_kernel<D, T>, a);
}

}  // namespace

#ifdef HKV_ATTN_TRACE
extern "C" int hkv_debug_set_step_trace(unsigned long long *buf) {
  return cudaMemcpyToSymbol(g_step_trace, &buf, sizeof(buf)) == cudaSuccess ? 0 : 7;
}
#endif

int step_tile_rows(int D, int dtype) {
  if (dtype == HKV_BF16) return D == 64 ? StepShape<64, __nv_bfloat16>::kTT : StepShape<128, __nv_bfloat16>::kTT;
  return D == 64 ? StepShape<64, float>::kTT : StepShape<128, float>::kTT;
}

cudaError_t step_prepare(int D, int dtype, int *ctas) {
  if (dtype == HKV_BF16)
    return D == 64 ? step_prepare_t<64, __nv_bfloat16>(ctas) : step_prepare_t<128, __nv_bfloat16>(ctas);
  return D == 64 ? step_prepare_t<64, float>(ctas) : step_prepare_t<128, float>(ctas);
}

cudaError_t launch_step(const AttnArgs &a, int D, int dtype, int grid, cudaStream_t s) {
  if (grid < 1 || grid > kAttnMaxGrid) return cudaErrorInvalidValue;
  if (dtype == HKV_BF16)
    return D == 64 ? step_launch_t<64, __nv_bfloat16>(a, grid, s)
                   : step_launch_t<128, __nv_bfloat16>(a, grid, s);
  return D == 64 ? step_launch_t<64, float>(a, grid, s) : step_launch_t<128, float>(a, grid, s);
}

}  // namespace hkv
