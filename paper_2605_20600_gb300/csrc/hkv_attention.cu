// Single-query decode attention over a ragged per-head KV cache (HeadKV,
// Eq. 1 applied to each head's retained tokens), optionally fused with the
// append of the step's new token.
//
// Two kernels per layer, chained with programmatic dependent launch:
//
// attention kernel (memory bound: every retained K/V byte is read once)
//  * split-K over the layer's total work, counted in tile slots: each head
//    is rounded up to whole tiles of TT rows, since under a saturated memory
//    system a tile costs one pipeline stage for one memory latency whatever
//    its fill. The concatenation of all heads' slots is split into
//    gridDim.x equal contiguous ranges, one per CTA, so local heads (short)
//    and global heads (long) load-balance; a range may cover the end of one
//    head, whole heads and the start of another;
//  * the prologue gives every thread a contiguous slice of the layer's heads
//    (one round of loads), a block scan locates each CTA's first head, and a
//    table of (offset, length, start) of the CTA's heads goes to shared
//    memory;
//  * warp-specialised pipeline: one producer warp streams K/V tiles of 10.5 KB
//    into shared memory with the TMA engine (1D cp.async.bulk) through NS
//    stages guarded by full/empty mbarriers, each with a description of its
//    tile; the query row of a head rides along with the head's first tile
//    and, fused, the new token's K/V with its last; an epilogue warp merges
//    the consumer warps' states of each head segment and writes the output
//    (a head wholly inside the piece) or a partial result (a split head)
//    while the consumers stream on. A CTA whose range starts inside a head
//    that began in the previous CTA's range records that head and how many
//    pieces it has; the head's first pieces go to slots of that CTA
//    boundary, the rest to the slot of the CTA that computed them;
//  * consumers take whole token rows with 16-byte lanes (a 256-byte bf16 row
//    is 16 lanes), a shuffle-xor tree per row for q.k, online softmax in the
//    log2 domain with fp32 accumulation;
//  * no fences or atomics;
//
//  * fused: the CTA whose range holds a head's last row appends the new
//    token (K/V row, position, query for the periodic update): nothing in
//    the launch reads them;
//
// finishing kernel (one-warp CTAs, after the attention kernel completes)
//  * a warp per CTA boundary merges the head split there from the pieces'
//    slots in index order, so the result does not depend on timing;
//  * fused: one lane per head advances the head's length and counters;
//
//  * programmatic dependent launch: every thread of either kernel waits for
//    the previous kernel of the stream (griddepcontrol.wait) before it reads
//    what that kernel writes or writes anything; with the prefetch flag the
//    attention prologue and the first NS tiles of old K/V rows go ahead of
//    that wait (HKV_ATTN_PRE_TILES of them: tiles in flight then delay the
//    previous finishing kernel, whose few loads are on the critical path);
//  * every wait on an mbarrier is bounded; one that runs out flags the
//    error and lets the CTA finish its control flow without the data, the
//    producer first waiting (bounded) for the bulk copies it armed.
#include <math.h>
#include <stdlib.h>

#include "hkv_attn_common.cuh"
#include "hkv_device.cuh"
#include "hkv_kernels.h"

namespace hkv {
namespace {

// Phase timestamps and counters per CTA for latency studies; compiled out by
// default.
#ifdef HKV_ATTN_TRACE
__device__ unsigned long long *g_trace = nullptr;  // [layer][kAttnMaxGrid][32], set by the tracer
#define HKV_TRACE_AT(slot) \
  g_trace[((size_t)(p.layer_base / p.nheads) * kAttnMaxGrid + blockIdx.x) * 32 + (slot)]
#define HKV_TRACE(slot)                              \
  do {                                               \
    if (g_trace) HKV_TRACE_AT(slot) = globaltimer(); \
  } while (0)
#define HKV_TRACE_ADD(slot, v)             \
  do {                                     \
    if (g_trace) HKV_TRACE_AT(slot) = (v); \
  } while (0)  // one writer per slot and launch: a plain store
#define HKV_CLOCK() globaltimer()
#else
#define HKV_TRACE(slot) \
  do {                  \
  } while (0)
#define HKV_TRACE_ADD(slot, v) \
  do {                         \
    (void)(v);                 \
  } while (0)
#define HKV_CLOCK() 0ull
#endif

constexpr int kTable = 32;  // heads of a CTA's range kept in smem

struct HeadTable {
  int h0;                   // first head of the table
  int n;                    // valid entries
  long long start[kTable];  // index (slot space) where head h0 + j starts
  long long off[kTable];    // arena offset of head h0 + j
  int vlen[kTable];         // virtual length (len + fused)
};

constexpr int kFirst = 1, kLast = 2, kDone = 4;

struct TileMeta {           // producer -> consumers, one per stage
  int h, n, flags;          // head, rows, kFirst | kLast | kDone
  int recent0;              // identification: rows from here on are among the
                            // head's newest w_loc - 1
  long long hs, he;         // the head's rows in the index space
};

struct SegMeta {            // consumers -> epilogue; h < 0: no more segments
  int h;
  long long hs, he;
};

template <bool FUSED>
struct HeadLookup {  // the table, else global memory
  const HeadTable &t;
  const AttnArgs &p;
  __device__ __forceinline__ int vlen(int h) const {
    const int j = h - t.h0;
    if (j >= 0 && j < t.n) return t.vlen[j];
    return h < p.nheads ? p.len[h] + (FUSED ? 1 : 0) : 0;
  }
  __device__ __forceinline__ long long off(int h) const {
    const int j = h - t.h0;
    if (j >= 0 && j < t.n) return t.off[j];
    return p.off[h];
  }
};

// what the producer must still add to a tile after its arena rows
struct Pending {
  int h, slot_new;
  bool first, has_new;
};

template <int D, typename T, bool FUSED, bool IDENT>
__global__ void __launch_bounds__(AttnShape<D, T>::kThreads, 2) attn_kernel(const AttnArgs p) {
  using S = AttnShape<D, T>;
  constexpr int kCW = S::kCW, kAttnThreads = S::kThreads;
  constexpr int LPR = S::kLPR, EPL = S::kEPL, RPW = S::kRPW, TT = S::kTT;
  constexpr int RB = S::kRB, NS = S::kNS;

  extern __shared__ __align__(128) unsigned char stages[];
  __shared__ uint64_t full[NS], empty[NS];
  __shared__ uint64_t epi_full, epi_free;   // hand-over of one segment's states
  // one segment's states: every row group of every consumer warp hands over
  // its own (the epilogue merges them), so no consumer spends a shuffle tree
  // on it
  constexpr int NST = kCW * RPW;
  static_assert(NST <= 32, "a lane of the epilogue per state");
  __shared__ __align__(16) float red_acc[NST][D];
  __shared__ float red_m[NST], red_l[NST];
  __shared__ float red_r[IDENT ? NST : 1];  // identification: mass of the newest rows
  __shared__ TileMeta meta[NS];
  __shared__ SegMeta seg;
  __shared__ HeadTable tab;
  __shared__ long long scan_scratch[33];
  __shared__ long long s_s0;
  __shared__ int s_h0, s_bad;
  __shared__ volatile int s_abort;
#ifdef HKV_ATTN_TRACE
  __shared__ unsigned long long t_issue[NS];
#endif

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nheads = p.nheads;
  const int G = gridDim.x;

  if (tid == 0) {
    HKV_TRACE(0);
#ifdef HKV_ATTN_TRACE
    if (g_trace) {
      unsigned smid;
      asm volatile("mov.u32 %0, %%smid;" : "=r"(smid));
      HKV_TRACE_AT(16) = smid;
    }
#endif
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kCW);
    }
    mbar_init(&epi_full, kCW);
    mbar_init(&epi_free, 1);
    fence_barrier_init();
    s_abort = 0;
    s_bad = 0;
    s_h0 = 0;
    s_s0 = 0;
  }
  // Without prefetch, wait for the previous kernel's writes first. With it,
  // the prologue and the first tiles of old K/V rows (which the caller
  // guarantees the previous kernel does not write) go ahead of the wait.
  if (!p.prefetch) pdl_wait();

  // ---- prologue: every thread takes a contiguous slice of the layer's heads
  // (every load of a head issued before any check uses one, so a group of
  // heads costs one round trip); a block scan gives each slice its first
  // slot.
  const int per = (nheads + kAttnThreads - 1) / kAttnThreads;
  const int h_lo = tid * per < nheads ? tid * per : nheads;
  const int h_hi = h_lo + per < nheads ? h_lo + per : nheads;
  long long mine = 0;
  int bad = 0;
  auto check = [&](int l, long long o, int cp, int lab, int nb) {
    if (l < 0 || o < 0 || o + l > p.arena_tokens) bad = HKV_ERR_BOUNDS;
    if (FUSED) {
      if (o + cp > p.arena_tokens) bad = HKV_ERR_BOUNDS;
      else if (l + 1 > cp) bad = bad ? bad : HKV_ERR_CAPACITY;
      else if (lab != HKV_DENSE && nb >= p.period)
        bad = bad ? bad : HKV_ERR_STATE;  // the periodic update is due first
      else if (IDENT && lab != HKV_DENSE)
        bad = bad ? bad : HKV_ERR_STATE;  // identification reads the dense cache's row order
    }
  };
#pragma unroll 4
  for (int h = h_lo; h < h_hi; ++h) {
    const int l = p.len[h];
    const long long o = p.off[h];
    if (FUSED)
      check(l, o, p.cap[h], p.label[p.layer_base + h], p.nbuf[p.layer_base + h]);
    else
      check(l, o, 0, 0, 0);
    mine += slot_len<TT>(l + (FUSED ? 1 : 0));
  }
  long long total;
  const long long slice_start = block_excl_scan<long long>(mine, scan_scratch, &total);
  if (bad) atomicMax(&s_bad, bad);
  __syncthreads();
  if (s_bad) {
    pdl_wait();
    if (blockIdx.x == 0 && tid == 0) {
      set_err(p.err, (uint32_t)s_bad);
      p.ctl->valid = 0;  // nothing for the finishing kernel to do
    }
    return;
  }
  // whole slots per CTA; rounding up leaves the last CTAs, which start
  // last, with less
  long long chunk = slot_len<TT>((total + G - 1) / G);
  if (chunk < S::kMinChunk) chunk = S::kMinChunk;
  const long long a = (long long)blockIdx.x * chunk;
  const long long b = a + chunk < total ? a + chunk : total;
  const bool st_active = a < total;
  const bool holds_a = st_active && mine > 0 && slice_start <= a && a < slice_start + mine;
  if (holds_a) {
    long long st = slice_start;
    for (int h = h_lo; h < h_hi; ++h) {
      const long long L = slot_len<TT>(p.len[h] + (FUSED ? 1 : 0));
      if (a < st + L) {
        s_h0 = h;
        s_s0 = st;
        break;
      }
      st += L;
    }
  }
  __syncthreads();
  if (warp == 0) {  // table of the heads from the CTA's first head on
    const int h0 = st_active ? s_h0 : 0;
    const int h = h0 + lane;
    const bool in = st_active && h < nheads;
    const int v = in ? p.len[h] + (FUSED ? 1 : 0) : 0;
    const long long L = slot_len<TT>(v);
    const long long incl = warp_incl_scan(L);
    tab.start[lane] = s_s0 + incl - L;
    tab.off[lane] = in ? p.off[h] : 0;
    tab.vlen[lane] = v;
    if (lane == 0) {
      tab.h0 = h0;
      tab.n = st_active ? (nheads - h0 < kTable ? nheads - h0 : kTable) : 0;
    }
  }
  __syncthreads();
  if (tid == 0) HKV_TRACE(1);
  const HeadLookup<FUSED> look{tab, p};

  // ---- producer state (warp 0, lane 0) ----------------------------------
  // A tile's old rows come from the arena; the query row (first tile of a
  // head in a piece) and the new token's K/V (fused, last tile of a head)
  // come from this step's inputs, which may be written by the previous
  // kernel.
  const bool producer = tid == 0;
  TileIter<TT> pit;
  pit.h = tab.h0;
  pit.hs = tab.start[0];
  pit.hl = tab.vlen[0];
  pit.g = st_active ? a : 0;
  pit.b = st_active ? b : 0;
  int issued = 0;
  // the arena rows are read once per step: evict them from L2 first
  const uint64_t stream_pol = producer ? l2_evict_first_policy() : 0;
  auto issue_old = [&](Pending &pd) {  // describe + expect + copy the arena rows
    const int stage = issued % NS;
#ifdef HKV_ATTN_TRACE
    t_issue[stage] = globaltimer();
#endif
    const long long ge = pit.tile_end();
    const long long he = pit.hs + pit.hl;
    const int r0 = (int)(pit.g - pit.hs), r1 = (int)(ge - pit.hs);   // head-local rows
    const int real = FUSED ? pit.hl - 1 : pit.hl;                    // rows in the arena
    const int n_old = (r1 < real ? r1 : real) - r0;
    unsigned char *dk = stages + stage * S::kStageBytes;
    pd.h = pit.h;
    pd.slot_new = real - r0;
    pd.first = pit.g == pit.hs || pit.g == a;
    pd.has_new = FUSED && r1 == pit.hl;
    TileMeta &mt = meta[stage];
    mt.h = pit.h;
    mt.n = (int)(ge - pit.g);
    mt.flags = (pd.first ? kFirst : 0) | (ge == (b < he ? b : he) ? kLast : 0);
    mt.hs = pit.hs;
    mt.he = he;
    if (IDENT) {
      const long long r0n = he - (p.w_loc - 1) - pit.g;  // first of the newest rows, tile-local
      mt.recent0 = r0n < 0 ? 0 : (int)(r0n < TT ? r0n : TT);
    }
    if (n_old > 0) {
      const uint32_t bytes = (uint32_t)n_old * RB;
      const long long row = look.off(pit.h) + r0;
      mbar_expect_tx(&full[stage], 2 * bytes);
      bulk_g2s_hint(dk, static_cast<const unsigned char *>(p.K) + row * RB, bytes, &full[stage],
                    stream_pol);
      bulk_g2s_hint(dk + TT * RB, static_cast<const unsigned char *>(p.V) + row * RB, bytes,
                    &full[stage], stream_pol);
    }
    pit.advance(look);
    ++issued;
  };
  auto issue_extra = [&](const Pending &pd, int stage) {  // inputs, then arrive
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
    for (; n_pre < (p.prefetch ? HKV_ATTN_PRE_TILES : NS) && !pit.done(); ++n_pre)
      issue_old(pre[n_pre]);

  if (p.prefetch) pdl_wait();  // the step's inputs are visible from here on
  if (tid == 0) HKV_TRACE(2);
  pdl_launch_dependents();
  // the launch passed its checks (the workspace is free: the previous
  // finishing kernel is done)
  if (blockIdx.x == 0 && tid == 0) p.ctl->valid = 1;
  // The head split at this CTA's boundary, if its first row lies in the
  // previous CTA's range: the finishing kernel merges its pieces (CTAs
  // k0 = blockIdx.x - 1 .. k0 + np - 1). Written by the epilogue warp, idle
  // until the first segment ends (the producer is on the critical path now).
  __shared__ int s_np;
  if (blockIdx.x > 0 && tid == (kCW + 1) * 32) {
    int4 r = make_int4(-1, 0, 0, 0);
    const long long hs = tab.start[0];
    if (st_active && hs < a && hs >= a - chunk) {
      const long long k0 = blockIdx.x - 1;
      const long long he = hs + tab.vlen[0];
      r = make_int4(tab.h0, (int)((he - 1) / chunk - k0 + 1), 0, 0);
    }
    p.rec[blockIdx.x] = r;
    // the inline slots of this boundary that no piece fills hold empty
    // pieces (maximum -inf, sum 0): the finishing kernel loads all of them
    s_np = r.x >= 0 ? r.y : 0;
  }

  if (warp == 0) {
    // ---- producer ----------------------------------------------------------
    if (producer) {
      unsigned long long t_wait = 0;
#pragma unroll
      for (int j = 0; j < NS; ++j)
        if (j < n_pre) issue_extra(pre[j], j);
      int armed = n_pre;  // tiles whose stage the producer has arrived on
      while (!pit.done()) {
        const int stage = issued % NS;
        // the consumers are done with the tile that used this stage before
        const unsigned long long tw = HKV_CLOCK();
        if (s_abort ||
            (issued >= NS && !mbar_wait(&empty[stage], (uint32_t)(issued / NS - 1) & 1u))) {
          s_abort = 1;
          set_err(p.err, HKV_ERR_TIMEOUT);
          break;
        }
        t_wait += HKV_CLOCK() - tw;
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
      if (s_abort) {
        // No bulk copy may land in shared memory after the CTA exits: wait
        // (bounded) for every armed stage that may still be in flight; a
        // stage reused after an empty-barrier wait is complete already.
        const int first = armed - NS > 0 ? armed - NS : 0;
        for (int t = first; t < armed; ++t) mbar_wait(&full[t % NS], (uint32_t)(t / NS) & 1u);
      }
      HKV_TRACE_ADD(13, t_wait);
    }
  } else if (warp <= kCW) {
    // ---- consumers ---------------------------------------------------------
    const int ctid = tid - 32, cw = warp - 1;
    const int grp = lane / LPR, col = lane % LPR;
    using M = LaneMath<T>;
    static_assert(M::kEPL == EPL, "lane mapping");
    typename M::Q q;
    float2 acc[EPL / 2];
    float m = -INFINITY, l = 0.f, lr = 0.f;  // lr: identification's newest-row mass
    int nseg = 0;
#pragma unroll
    for (int e = 0; e < EPL / 2; ++e) acc[e] = make_float2(0.f, 0.f);

    unsigned long long t_full = 0, t_stall = 0, t_lat = 0;
    long long c_comp = 0, c_last = 0;
    int n_tiles = 0;
    for (int tile = 0;; ++tile) {
      const int stage = tile % NS;
      const unsigned long long tw = HKV_CLOCK();
      if (!s_abort && !mbar_wait(&full[stage], (uint32_t)(tile / NS) & 1u)) {
        s_abort = 1;
        set_err(p.err, HKV_ERR_TIMEOUT);
      }
      if (tile > 0) t_full += HKV_CLOCK() - tw;
#ifdef HKV_ATTN_TRACE
      const long long c_t0 = clock64();
      if (!s_abort && !(meta[stage].flags & kDone)) t_lat += HKV_CLOCK() - t_issue[stage];
#endif
      if (s_abort) break;
      const int flags = meta[stage].flags;
      if (flags & kDone) break;
      if (tile == 0 && ctid == 0) HKV_TRACE(3);
      ++n_tiles;
      const int n = meta[stage].n;
      const unsigned char *Ks = stages + stage * S::kStageBytes;
      const unsigned char *Vs = Ks + TT * RB;
      if (flags & kFirst) {  // first tile of this head in this piece
        M::load_q(q, *reinterpret_cast<const uint4 *>(Vs + TT * RB + col * 16), p.qscale);
#pragma unroll
        for (int e = 0; e < EPL / 2; ++e) acc[e] = make_float2(0.f, 0.f);
        m = -INFINITY;
        l = 0.f;
        lr = 0.f;
      }
      const int recent0 = IDENT ? meta[stage].recent0 : 0;

      float sc[S::kSteps];
#pragma unroll
      for (int st = 0; st < S::kSteps; ++st) {
        const int r = st * (kCW * RPW) + cw * RPW + grp;
        float dot = 0.f;
        if (r < n) dot = M::dot(q, *reinterpret_cast<const uint4 *>(Ks + r * RB + col * 16));
#pragma unroll
        for (int o = LPR / 2; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xFFFFFFFFu, dot, o);
        sc[st] = r < n ? M::score(dot, p.qscale) : -INFINITY;
      }
      float mt = sc[0];
#pragma unroll
      for (int st = 1; st < S::kSteps; ++st) mt = fmaxf(mt, sc[st]);
      const float mn = fmaxf(m, mt);
      if (mn != -INFINITY) {
        const float corr = exp2f(m - mn);
        l *= corr;
        if (IDENT) lr *= corr;
#pragma unroll
        for (int e = 0; e < EPL / 2; ++e) acc[e] = __fmul2_rn(acc[e], make_float2(corr, corr));
#pragma unroll
        for (int st = 0; st < S::kSteps; ++st) {
          const int r = st * (kCW * RPW) + cw * RPW + grp;
          if (r < n) {
            const float pr = exp2f(sc[st] - mn);
            l += pr;
            if (IDENT && r >= recent0) lr += pr;
            M::add_v(acc, *reinterpret_cast<const uint4 *>(Vs + r * RB + col * 16), pr);
          }
        }
        m = mn;
      }
#ifdef HKV_ATTN_TRACE
      const long long c_t1 = clock64();
      c_comp += c_t1 - c_t0;
#endif
      if (flags & kLast) {  // last tile of this head in this piece: hand it over
        SegMeta sm;
        if (cw == 0 && lane == 0) {
          sm.h = meta[stage].h;
          sm.hs = meta[stage].hs;
          sm.he = meta[stage].he;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[stage]);  // this warp is done with the stage
        // the epilogue is done with the previous segment's states
        const unsigned long long tw = HKV_CLOCK();
        if (nseg > 0 && !s_abort && !mbar_wait(&epi_free, (uint32_t)(nseg - 1) & 1u)) {
          s_abort = 1;
          set_err(p.err, HKV_ERR_TIMEOUT);
        }
        t_stall += HKV_CLOCK() - tw;
        {  // this row group's state
          const int si = cw * RPW + grp;
          float2 *dst = reinterpret_cast<float2 *>(&red_acc[si][col * EPL]);
#pragma unroll
          for (int e = 0; e < EPL / 2; ++e) dst[e] = acc[e];
          if (col == 0) {
            red_m[si] = m;
            red_l[si] = l;
            if (IDENT) red_r[si] = lr;
          }
        }
        if (cw == 0 && lane == 0) seg = sm;
        __syncwarp();
        if (lane == 0) mbar_arrive(&epi_full);
        ++nseg;
#ifdef HKV_ATTN_TRACE
        c_last += clock64() - c_t1;
#endif
      } else {
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[stage]);  // this warp is done with the stage
      }
    }
    if (ctid == 0) HKV_TRACE(4);
    if (ctid == 0) HKV_TRACE_ADD(12, t_full);
    if (ctid == 0) HKV_TRACE_ADD(11, t_stall);
    if (ctid == 0) HKV_TRACE_ADD(17, n_tiles);
    if (ctid == 0) HKV_TRACE_ADD(24, c_comp);
    if (ctid == 0) HKV_TRACE_ADD(25, c_last);
    if (ctid == 0) HKV_TRACE_ADD(26, t_lat);
    // tell the epilogue there is nothing more
    if (nseg > 0 && !s_abort && !mbar_wait(&epi_free, (uint32_t)(nseg - 1) & 1u)) {
      s_abort = 1;
      set_err(p.err, HKV_ERR_TIMEOUT);
    }
    if (cw == 0 && lane == 0) seg.h = -1;
    __syncwarp();
    if (lane == 0) mbar_arrive(&epi_full);
  } else {
    // ---- epilogue: finish each head segment the consumers hand over --------
    // A lane owns CPL consecutive output channels, so each of its stores of
    // an output row or a partial result is one vector access.
    constexpr int CPL = D / 32;
    using V = Vec<CPL>;
    constexpr int PS = attn_part_floats(D);  // floats per partial slot
    if (blockIdx.x > 0) {
      __syncwarp();
      const int np0 = s_np;  // written by lane 0 of this warp above
      float z[CPL];
#pragma unroll
      for (int c = 0; c < CPL; ++c) z[c] = 0.f;
      for (int j = np0; j < kAttnInlinePieces; ++j) {
        float *pp = p.part + ((size_t)blockIdx.x * kAttnInlinePieces + j) * PS;
        V::st(pp + CPL * lane, z);
        if (lane == 0) {
          pp[D] = -INFINITY;
          pp[D + 1] = 0.f;
          pp[D + 2] = 0.f;
        }
      }
    }
    unsigned long long t_ew = 0, t_eb = 0, t_e1 = HKV_CLOCK();
    int k_segs = 0;
    for (int k = 0;; ++k, ++k_segs) {
      const unsigned long long t_e0 = HKV_CLOCK();
      if (k > 0) t_eb += t_e0 - t_e1;
      if (!s_abort && !mbar_wait(&epi_full, (uint32_t)k & 1u)) {
        s_abort = 1;
        set_err(p.err, HKV_ERR_TIMEOUT);
      }
      t_e1 = HKV_CLOCK();
      if (k > 0) t_ew += t_e1 - t_e0;
      if (s_abort) break;
      const int h = seg.h;
      if (h < 0) break;
      const long long hs = seg.hs, he = seg.he;
      // merge the row-group states: lane s < NST weighs state s
      const float ms = lane < NST ? red_m[lane] : -INFINITY;
      float mx = ms;
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
      const float ws = ms == -INFINITY ? 0.f : exp2f(ms - mx);
      float L = lane < NST ? red_l[lane] * ws : 0.f;
      float LR = IDENT && lane < NST ? red_r[lane] * ws : 0.f;
#pragma unroll
      for (int o = 16; o >= 1; o >>= 1) {
        L += __shfl_xor_sync(0xFFFFFFFFu, L, o);
        if (IDENT) LR += __shfl_xor_sync(0xFFFFFFFFu, LR, o);
      }
      float A[CPL];
#pragma unroll
      for (int c = 0; c < CPL; ++c) A[c] = 0.f;
#pragma unroll
      for (int si = 0; si < NST; ++si) {
        const float sw = __shfl_sync(0xFFFFFFFFu, ws, si);
        float r[CPL];
        V::lds(&red_acc[si][CPL * lane], r);
#pragma unroll
        for (int c = 0; c < CPL; ++c) A[c] = fmaf(r[c], sw, A[c]);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&epi_free);  // the consumers may reuse the slot
      if (hs >= a && he <= b) {  // the whole head is in this CTA's range
#pragma unroll
        for (int c = 0; c < CPL; ++c) A[c] /= L;
        V::st(p.out + (size_t)h * D + CPL * lane, A);
        // Sec. 4 Step 2: local iff the newest w_loc - 1 tokens hold a share
        // tau of the attention
        if (IDENT && lane == 0)
          p.label_out[p.layer_base + h] = LR >= p.tau * L ? HKV_LOCAL : HKV_GLOBAL;
      } else {  // piece j of the head split at boundary k0 + 1
        const long long k0 = hs / chunk;
        const int j = (int)(blockIdx.x - k0);
        float *pp = j < kAttnInlinePieces
                        ? p.part + ((size_t)(k0 + 1) * kAttnInlinePieces + j) * PS
                        : p.over + (size_t)blockIdx.x * PS;
        V::st(pp + CPL * lane, A);
        if (lane == 0) {
          pp[D] = mx;
          pp[D + 1] = L;
          if (IDENT) pp[D + 2] = LR;
        }
      }
      // Fused: the CTA whose range holds the head's last row appends the new
      // token (K/V row at index len, its position, q into the ring of the
      // periodic update). Nothing in this launch reads them; the finishing
      // kernel advances the counters once every CTA is done.
      if (FUSED && he <= b) {
        const int i = p.layer_base + h;
        const int len = (int)(he - hs) - 1;
        const long long row = look.off(h) + len;
        const int nt = p.ntok[i];
        for (int c = lane; c < RB / 16; c += 32) {
          const uint4 kx = reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(p.k_new) + (size_t)h * RB)[c];
          const uint4 vx = reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(p.v_new) + (size_t)h * RB)[c];
          const uint4 qx = reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(p.q) + (size_t)h * RB)[c];
          reinterpret_cast<uint4 *>(static_cast<unsigned char *>(p.K) + row * RB)[c] = kx;
          reinterpret_cast<uint4 *>(static_cast<unsigned char *>(p.V) + row * RB)[c] = vx;
          reinterpret_cast<uint4 *>(static_cast<unsigned char *>(p.qbuf) +
                                    ((size_t)i * p.period + nt % p.period) * RB)[c] = qx;
        }
        if (lane == 0) p.pos[row] = p.n_cond + nt;
      }
    }
    if (lane == 0) HKV_TRACE(5);
    if (lane == 0) HKV_TRACE_ADD(14, t_eb);
    if (lane == 0) HKV_TRACE_ADD(9, k_segs);
    if (lane == 0) HKV_TRACE_ADD(15, t_ew);
  }
  if (tid == 0) HKV_TRACE(6);
}

// One-warp CTAs. Warp w advances the counters of heads 32w .. 32w + 31, one
// lane per head (fused; plain attention writes zeros for empty heads), and
// merges the head split at CTA boundary k = w + 1, if any, from its pieces in
// index order, so the result does not depend on timing. The record of that
// head and the boundary's inline slots (its first pieces, or empty pieces
// the attention kernel wrote there) load in the same round as the counters:
// a head of at most kAttnInlinePieces pieces costs one round trip to memory.
template <int D, typename T, bool FUSED, bool IDENT>
__global__ void __maxnreg__(IDENT ? kFinishRegs + 16 : kFinishRegs)
    finish_kernel(const AttnArgs p) {
  constexpr int CPL = D / 32;
  using V = Vec<CPL>;
  constexpr int PS = attn_part_floats(D);
  constexpr int NI = kAttnInlinePieces;  // pieces per batch (the first: inline)
  // Let the next kernel (the next layer's attention) start its prologue now;
  // it waits for this kernel before it reads anything written here.
  HKV_TRACE(20);
  pdl_launch_dependents();
  pdl_wait();  // the attention kernel is complete
  HKV_TRACE(21);
  const int lane = threadIdx.x & 31;
  const int w = blockIdx.x * (kFinishThreads / 32) + (threadIdx.x >> 5);
  const int G = p.grid;
  const int valid = p.ctl->valid;
  const int h = 32 * w + lane;
  const bool hin = h < p.nheads;
  const int i = p.layer_base + h;
  int len = 0, nt = 0, nb = 0;
  bool dense = true;
  if (hin) {
    len = p.len[h];
    if (FUSED) {
      nt = p.ntok[i];
      nb = p.nbuf[i];
      dense = p.label[i] == HKV_DENSE;
    }
  }
  const int k = w + 1;  // the boundary between CTAs k - 1 and k
  int4 rc = make_int4(-1, 0, 0, 0);
  float iv[NI][CPL];
  float im[NI], il[NI];  // maxima and sums of the inline pieces (every lane)
  float ir[IDENT ? NI : 1];  // identification: their newest-row masses
#pragma unroll
  for (int u = 0; u < NI; ++u) {
    im[u] = -INFINITY;
    il[u] = 0.f;
    if (IDENT) ir[u] = 0.f;
#pragma unroll
    for (int c = 0; c < CPL; ++c) iv[u][c] = 0.f;
  }
  const float *inl = p.part + (size_t)k * NI * PS;
  if (k < G) {
    rc = __ldcg(p.rec + k);
#pragma unroll
    for (int u = 0; u < NI; ++u) {
      V::ldcg(inl + (size_t)u * PS + CPL * lane, iv[u]);
      im[u] = __ldcg(inl + (size_t)u * PS + D);
      il[u] = __ldcg(inl + (size_t)u * PS + D + 1);
      if (IDENT) ir[u] = __ldcg(inl + (size_t)u * PS + D + 2);
    }
  }
#ifdef HKV_ATTN_TRACE
  if (g_trace && lane == 0) HKV_TRACE_AT(27) = rc.x >= 0 ? rc.y : 0;
  if (g_trace && lane == 0 &&
      (len + nt + nb + rc.x + valid + (int)(im[0] + il[NI - 1] + iv[NI - 1][0] + iv[0][0])) != 0x7fffffff)
    HKV_TRACE_AT(23) = globaltimer();  // the loads are back
#endif
  if (valid) {  // else the attention launch failed its checks
    if (FUSED && hin) {  // the new token joined the head in the attention kernel
      p.len[h] = len + 1;
      p.ntok[i] = nt + 1;
      if (!dense) p.nbuf[i] = nb + 1;
    }
    if (!FUSED && hin && len == 0) {  // an empty head has no tiles: zeros
      float4 *o = reinterpret_cast<float4 *>(p.out + (size_t)h * D);
#pragma unroll 4
      for (int c = 0; c < D / 4; ++c) o[c] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  if (valid && rc.x >= 0 && rc.y <= NI) {
    // at most NI pieces, all inline (the slots past the last piece hold empty
    // pieces: weight 0): every lane merges them in piece order with no
    // exchange, the largest maximum first, then the weighted sums
    float gm = im[0];
#pragma unroll
    for (int u = 1; u < NI; ++u) gm = fmaxf(gm, im[u]);
    float GL = 0.f, GR = 0.f, GA[CPL];
#pragma unroll
    for (int c = 0; c < CPL; ++c) GA[c] = 0.f;
#pragma unroll
    for (int u = 0; u < NI; ++u) {
      const float wu = im[u] == -INFINITY ? 0.f : exp2f(im[u] - gm);
      GL += il[u] * wu;
      if (IDENT) GR += ir[u] * wu;
#pragma unroll
      for (int c = 0; c < CPL; ++c) GA[c] = fmaf(iv[u][c], wu, GA[c]);
    }
#pragma unroll
    for (int c = 0; c < CPL; ++c) GA[c] /= GL;
    V::st(p.out + (size_t)rc.x * D + CPL * lane, GA);
    if (IDENT && lane == 0)  // Sec. 4 Step 2, as in the attention kernel
      p.label_out[p.layer_base + rc.x] = GR >= p.tau * GL ? HKV_LOCAL : HKV_GLOBAL;
  } else if (valid && rc.x >= 0) {
    const int hh = rc.x, np = rc.y;
    // piece j >= NI: the overflow slot of the CTA that computed it
    auto over = [&](int j) { return p.over + (size_t)(k - 1 + j) * PS; };
    float m0 = -INFINITY, l0 = 0.f, r0 = 0.f;  // piece `lane`
#pragma unroll
    for (int u = 0; u < NI; ++u)
      if (lane == u) {
        m0 = im[u];
        l0 = il[u];
        if (IDENT) r0 = ir[u];
      }
    if (lane >= NI && lane < np) {
      m0 = __ldcg(over(lane) + D);
      l0 = __ldcg(over(lane) + D + 1);
      if (IDENT) r0 = __ldcg(over(lane) + D + 2);
    }
    // Merge in piece (index) order: the maximum first, then the weighted sums
    // (inline slots past the last piece hold empty pieces: weight 0).
    float gm = m0;
    for (int j = lane + 32; j < np; j += 32) gm = fmaxf(gm, __ldcg(over(j) + D));
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) gm = fmaxf(gm, __shfl_xor_sync(0xFFFFFFFFu, gm, o));
    float GL = 0.f, GR = 0.f, GA[CPL];
#pragma unroll
    for (int c = 0; c < CPL; ++c) GA[c] = 0.f;
    for (int j0 = 0; j0 < np; j0 += 32) {
      float mj = m0, lj = l0, rj = r0;
      if (j0 > 0) {
        const int j = j0 + lane;
        mj = -INFINITY;
        lj = rj = 0.f;
        if (j < np) {
          mj = __ldcg(over(j) + D);
          lj = __ldcg(over(j) + D + 1);
          if (IDENT) rj = __ldcg(over(j) + D + 2);
        }
      }
      // weight of piece j0 + lane (zero past the last piece)
      const float wj = mj == -INFINITY ? 0.f : exp2f(mj - gm);
      const float lw = lj * wj;
      const float rw = IDENT ? rj * wj : 0.f;
      const int cnt = np - j0 < 32 ? np - j0 : 32;
      for (int t0 = 0; t0 < cnt; t0 += NI) {
        float v[NI][CPL];
        if (j0 == 0 && t0 == 0) {
#pragma unroll
          for (int u = 0; u < NI; ++u)
#pragma unroll
            for (int c = 0; c < CPL; ++c) v[u][c] = iv[u][c];
        } else {
#pragma unroll
          for (int u = 0; u < NI; ++u) {
            if (j0 + t0 + u < np) {
              V::ldcg(over(j0 + t0 + u) + CPL * lane, v[u]);
            } else {
#pragma unroll
              for (int c = 0; c < CPL; ++c) v[u][c] = 0.f;
            }
          }
        }
#pragma unroll
        for (int u = 0; u < NI; ++u) {
          const float wu = __shfl_sync(0xFFFFFFFFu, wj, t0 + u);
          GL += __shfl_sync(0xFFFFFFFFu, lw, t0 + u);
          if (IDENT) GR += __shfl_sync(0xFFFFFFFFu, rw, t0 + u);
          if (j0 + t0 + u < np)
#pragma unroll
            for (int c = 0; c < CPL; ++c) GA[c] = fmaf(v[u][c], wu, GA[c]);
        }
      }
    }
#pragma unroll
    for (int c = 0; c < CPL; ++c) GA[c] /= GL;
    V::st(p.out + (size_t)hh * D + CPL * lane, GA);
    if (IDENT && lane == 0)
      p.label_out[p.layer_base + hh] = GR >= p.tau * GL ? HKV_LOCAL : HKV_GLOBAL;
  }
  HKV_TRACE(22);
}

template <int D, typename T>
size_t smem_bytes() {
  return (size_t)AttnShape<D, T>::kNS * AttnShape<D, T>::kStageBytes;
}

template <int D, typename T, bool F, bool I>
cudaError_t prepare_t(int *ctas) {
  const size_t smem = smem_bytes<D, T>();
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<D, T, F, I>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas, attn_kernel<D, T, F, I>,
                                                       AttnShape<D, T>::kThreads, smem);
}

template <int D, typename T>
cudaError_t prepare_all(int *ctas) {
  int a = 0, b = 0, c = 0;
  cudaError_t e = prepare_t<D, T, false, false>(&a);
  if (e == cudaSuccess) e = prepare_t<D, T, true, false>(&b);
  if (e == cudaSuccess) e = prepare_t<D, T, true, true>(&c);
  *ctas = a < b ? a : b;
  if (c < *ctas) *ctas = c;
  if (*ctas > HKV_ATTN_MAX_CTAS_PER_SM) *ctas = HKV_ATTN_MAX_CTAS_PER_SM;
  return e;
}

template <typename K>
cudaError_t launch_pdl(K kernel, int grid, int threads, size_t smem, const AttnArgs &a,
                       cudaStream_t s) {
  static const bool pdl = getenv("HKV_NO_PDL") == nullptr;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, a);
}

template <int D, typename T, bool F, bool I>
cudaError_t launch_both(const AttnArgs &a, int grid, cudaStream_t s) {
  cudaError_t e = launch_pdl(attn_kernel<D, T, F, I>, grid, AttnShape<D, T>::kThreads,
                             smem_bytes<D, T>(), a, s);
  if (e != cudaSuccess) return e;
  // a warp for every 32 heads and for every CTA boundary
  int warps = (a.nheads + 31) / 32;
  if (warps < grid - 1) warps = grid - 1;
  if (warps < 1) warps = 1;
  const int fgrid = (warps + kFinishThreads / 32 - 1) / (kFinishThreads / 32);
  return launch_pdl(finish_kernel<D, T, F, I>, fgrid, kFinishThreads, 0, a, s);
}

template <int D, typename T>
cudaError_t launch_t(AttnArgs a, int grid, bool fused, bool identify, cudaStream_t s) {
  a.grid = grid;
  if (!fused) return launch_both<D, T, false, false>(a, grid, s);
  return identify ? launch_both<D, T, true, true>(a, grid, s)
                  : launch_both<D, T, true, false>(a, grid, s);
}

}  // namespace

#ifdef HKV_ATTN_TRACE
// tracer builds only: where the phase timestamps go
extern "C" int hkv_debug_set_trace(unsigned long long *buf) {
  return cudaMemcpyToSymbol(g_trace, &buf, sizeof(buf)) == cudaSuccess ? 0 : 7;
}
#endif

size_t attention_smem_bytes(int D, int dtype) {
  if (dtype == HKV_BF16) return D == 64 ? smem_bytes<64, __nv_bfloat16>() : smem_bytes<128, __nv_bfloat16>();
  return D == 64 ? smem_bytes<64, float>() : smem_bytes<128, float>();
}

cudaError_t attention_prepare(int D, int dtype, int *ctas) {
  if (dtype == HKV_BF16) return D == 64 ? prepare_all<64, __nv_bfloat16>(ctas) : prepare_all<128, __nv_bfloat16>(ctas);
  return D == 64 ? prepare_all<64, float>(ctas) : prepare_all<128, float>(ctas);
}

cudaError_t launch_attention(const AttnArgs &a, int D, int dtype, int grid, bool fused,
                             bool identify, cudaStream_t s) {
  if (grid < 1 || grid > kAttnMaxGrid) return cudaErrorInvalidValue;
  if (dtype == HKV_BF16)
    return D == 64 ? launch_t<64, __nv_bfloat16>(a, grid, fused, identify, s)
                   : launch_t<128, __nv_bfloat16>(a, grid, fused, identify, s);
  return D == 64 ? launch_t<64, float>(a, grid, fused, identify, s)
                 : launch_t<128, float>(a, grid, fused, identify, s);
}

}  // namespace hkv
