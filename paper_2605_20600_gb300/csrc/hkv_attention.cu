// Single-query decode attention over a ragged per-head KV cache (HeadKV,
// Eq. 1 applied to each head's retained tokens), optionally fused with the
// append of the step's new token.
//
// Design (GB300, memory bound: every retained K/V byte is read once):
//  * split-K over the layer's TOTAL token count: the concatenation of all
//    heads' live tokens is cut into gridDim.x equal contiguous ranges, so
//    local heads (short) and global heads (long) load-balance exactly; a
//    range may cover the end of one head, whole heads, and the start of
//    another;
//  * the prologue gives every thread a contiguous slice of the layer's
//    heads (one round of loads), a block scan finds the CTA's first head,
//    and a table of the next heads' (offset, length, start) goes to shared
//    memory;
//  * warp-specialised pipeline: one producer warp streams K/V tiles of 7 KB
//    into shared memory with the TMA engine (1D cp.async.bulk) through
//    NS stages guarded by full/empty mbarriers; the query row of a head rides
//    along with the head's first tile; consumer warps never wait on the
//    producer's issue work; an epilogue warp finishes each head segment
//    (merge of the consumer warps' states, output or partial result,
//    combine) while the consumers stream on;
//  * consumers take whole token rows with 16-byte lanes (a 256-byte bf16 row
//    is 16 lanes), a shuffle-xor tree per row for q.k, online softmax in the
//    log2 domain with fp32 accumulation;
//  * a head split across CTAs is combined by the last CTA to arrive (per-head
//    atomic counter, no spinning); partials are merged in CTA order, so the
//    result does not depend on arrival order;
//  * fused append: the head's virtual length is len + 1, the new token's K/V
//    come straight from the step's input rows, the CTA that finishes a head
//    writes that head's new row, and the last CTA of the grid (grid-wide
//    arrival counter) advances every head's counters once no CTA can still
//    be reading them;
//  * programmatic dependent launch: every thread waits for the previous
//    kernel of the stream (griddepcontrol.wait) before it reads the step's
//    inputs or writes anything; with the prefetch flag the prologue and the
//    first NS tiles of old K/V rows go ahead of that wait;
//  * every wait on an mbarrier is bounded; one that runs out flags the
//    error and lets the CTA finish its control flow without the data.
#include <math.h>
#include <stdlib.h>

#include "hkv_device.cuh"
#include "hkv_kernels.h"

namespace hkv {
namespace {

// Tuning knobs (compile time): bytes of K per pipeline stage, stages, and
// a cap on resident CTAs per SM used to size the grid.
#ifndef HKV_ATTN_TILE_BYTES
#define HKV_ATTN_TILE_BYTES 7168
#endif
#ifndef HKV_ATTN_STAGES
#define HKV_ATTN_STAGES 4
#endif
#ifndef HKV_ATTN_MAX_CTAS_PER_SM
#define HKV_ATTN_MAX_CTAS_PER_SM 32
#endif

constexpr int kCW = kAttnConsumerWarps;

// Phase timestamps per CTA for latency studies; compiled out by default.
#ifdef HKV_ATTN_TRACE
__device__ unsigned long long *g_trace = nullptr;  // [layer][kAttnMaxGrid][8], set by the tracer
#define HKV_TRACE(slot)                                                  \
  do {                                                                   \
    if (g_trace)                                                         \
      g_trace[((size_t)(p.layer_base / p.nheads) * kAttnMaxGrid + blockIdx.x) * 8 + (slot)] = \
          globaltimer();                                                 \
  } while (0)
#else
#define HKV_TRACE(slot) \
  do {                  \
  } while (0)
#endif

template <int D, typename T>
struct AttnShape {
  static constexpr int kES = sizeof(T);
  static constexpr int kRB = D * kES;             // bytes per token row
  static constexpr int kLPR = kRB / 16;           // lanes per row
  static constexpr int kEPL = 16 / kES;           // elements per lane
  static constexpr int kRPW = 32 / kLPR;          // rows per warp step
  static constexpr int kTT = HKV_ATTN_TILE_BYTES / kRB;   // rows per tile
  static constexpr int kSteps = kTT / (kCW * kRPW);
  static constexpr int kNS = HKV_ATTN_STAGES;     // pipeline stages
  static constexpr int kStageBytes = 2 * kTT * kRB + kRB;   // K, V, q row
  static constexpr int kMinChunk = 2 * kTT;       // fewest tokens per CTA
  static_assert(kLPR >= 1 && kLPR <= 32 && 32 % kLPR == 0, "row mapping");
  static_assert(kSteps >= 1 && kTT % (kCW * kRPW) == 0, "tile mapping");
  static_assert(D <= kCW * 32, "one consumer thread per output channel");
  static_assert(kStageBytes % 16 == 0, "TMA alignment");
};

constexpr int kTable = 32;  // heads whose (offset, length, start) sit in smem

struct HeadTable {
  int h0;                   // first head of the CTA's range
  int n;                    // valid entries
  int covers;               // the entries cover the CTA's whole range
  long long start[kTable];  // global token index where head h0 + j starts
  long long off[kTable];    // arena offset of head h0 + j
  int vlen[kTable];         // virtual length (len + fused)
  int ntok[kTable];         // image tokens appended so far (fused)
};

__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <bool FUSED>
struct HeadLookup {
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

// Walks the tiles of one CTA's token range [g, b) head by head.
struct TileIter {
  int h;         // current head (layer-local index)
  int hl;        // its (virtual) length
  long long hs;  // global token index where head h starts
  long long g;   // start of the current tile
  long long b;   // end of the CTA's range

  __device__ __forceinline__ bool done() const { return g >= b; }
  __device__ __forceinline__ long long tile_end(int tt) const {
    long long e = g + tt;
    const long long he = hs + hl;
    if (e > he) e = he;
    if (e > b) e = b;
    return e;
  }
  template <class L>
  __device__ __forceinline__ void advance(int tt, const L &look) {
    g = tile_end(tt);
    if (g >= b) return;
    while (g >= hs + hl) {  // next head holding token g (skips empty heads)
      hs += hl;
      ++h;
      hl = look.vlen(h);
    }
  }
};

// what the producer must still add to a tile after its arena rows
struct Pending {
  int h, slot_new;
  bool first, has_new;
};

template <int D, typename T, bool FUSED>
__global__ void __launch_bounds__(kAttnThreads, 3) attn_kernel(const AttnArgs p) {
  using S = AttnShape<D, T>;
  constexpr int LPR = S::kLPR, EPL = S::kEPL, RPW = S::kRPW, TT = S::kTT;
  constexpr int RB = S::kRB, NS = S::kNS;

  extern __shared__ __align__(128) unsigned char stages[];
  __shared__ uint64_t full[NS], empty[NS];
  __shared__ uint64_t epi_full, epi_free;   // hand-over of one segment's states
  __shared__ float red_acc[kCW][D];
  __shared__ float red_m[kCW], red_l[kCW];
  __shared__ int seg_h, seg_final;
  __shared__ long long seg_hs, seg_he;
  __shared__ HeadTable tab;
  __shared__ long long scan_scratch[33];
  __shared__ long long s_s0;
  __shared__ int s_h0, s_bad, s_last;
  __shared__ volatile int s_abort;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nheads = p.nheads;

  if (tid == 0) {
    HKV_TRACE(0);
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kCW);
    }
    mbar_init(&epi_full, kCW);
    mbar_init(&epi_free, 1);
    fence_barrier_init();
    s_abort = 0;
  }
  // Without prefetch, wait for the previous kernel's writes first. With it,
  // the prologue and the first tiles of old K/V rows (which the caller
  // guarantees the previous kernel does not write) go ahead of the wait.
  if (!p.prefetch) pdl_wait();

  // ---- prologue: every thread takes a contiguous slice of the layer's heads
  // (all of its loads in flight at once), a block scan gives each slice its
  // first token, and the slice holding token a names the CTA's first head.
  const int per = (nheads + kAttnThreads - 1) / kAttnThreads;
  const int h_lo = tid * per < nheads ? tid * per : nheads;
  const int h_hi = h_lo + per < nheads ? h_lo + per : nheads;
  long long mine = 0;
  int bad = 0;
#pragma unroll 4
  for (int h = h_lo; h < h_hi; ++h) {
    const int l = p.len[h];
    const long long o = p.off[h];
    if (l < 0 || o < 0 || o + l > p.arena_tokens) bad = HKV_ERR_BOUNDS;
    if (FUSED) {
      const int cp = p.cap[h];
      if (o + cp > p.arena_tokens) bad = HKV_ERR_BOUNDS;
      else if (l + 1 > cp) bad = bad ? bad : HKV_ERR_CAPACITY;
      else if (p.label[p.layer_base + h] != HKV_DENSE && p.nbuf[p.layer_base + h] >= p.period)
        bad = bad ? bad : HKV_ERR_STATE;  // the periodic update is due first
    }
    mine += l + (FUSED ? 1 : 0);
  }
  long long total;
  const long long slice_start = block_excl_scan<long long>(mine, scan_scratch, &total);
  if (tid == 0) s_bad = 0;
  __syncthreads();
  if (bad) atomicMax(&s_bad, bad);
  __syncthreads();
  if (s_bad) {
    pdl_wait();
    if (blockIdx.x == 0 && tid == 0) set_err(p.err, (uint32_t)s_bad);
    return;
  }
  long long chunk = (total + gridDim.x - 1) / gridDim.x;
  if (chunk < S::kMinChunk) chunk = S::kMinChunk;
  const long long a = (long long)blockIdx.x * chunk;
  const long long b = a + chunk < total ? a + chunk : total;
  const bool active = a < total;
  if (active && mine > 0 && slice_start <= a && a < slice_start + mine) {
    long long st = slice_start;
    for (int h = h_lo; h < h_hi; ++h) {
      const long long L = p.len[h] + (FUSED ? 1 : 0);
      if (a < st + L) {
        s_h0 = h;
        s_s0 = st;
        break;
      }
      st += L;
    }
  }
  __syncthreads();
  if (active && warp == 0) {  // table of the heads from h0 on
    const int h0 = s_h0;
    const int h = h0 + lane;
    const long long L = h < nheads ? p.len[h] + (FUSED ? 1 : 0) : 0;
    const long long incl = warp_incl_scan(L);
    tab.start[lane] = s_s0 + incl - L;
    tab.off[lane] = h < nheads ? p.off[h] : 0;
    tab.vlen[lane] = (int)L;
    tab.ntok[lane] = (FUSED && h < nheads) ? p.ntok[p.layer_base + h] : 0;
    const int n = nheads - h0 < kTable ? nheads - h0 : kTable;
    const long long end = __shfl_sync(0xFFFFFFFFu, s_s0 + incl, n - 1);
    if (lane == 0) {
      tab.h0 = h0;
      tab.n = n;
      tab.covers = end >= b;
    }
  }
  __syncthreads();
  // Fused: a CTA whose heads all sit in the table reads no length, position
  // counter or buffer count after this point, so it can count itself on the
  // grid counter as soon as the previous kernel is done (the counter lives in
  // the shared workspace); the last CTA to count advances the counters. The
  // other CTAs count at the end.
  const bool early = FUSED && (!active || tab.covers);

  if (tid == 0) HKV_TRACE(1);
  auto grid_arrive = [&]() {  // block-wide; called after the wait
    __syncthreads();
    if (tid == 0) {
      __threadfence();
      s_last = atomicAdd(p.gcnt, 1) == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (s_last) {
      __threadfence();
      for (int h = tid; h < nheads; h += kAttnThreads) {
        const int i = p.layer_base + h;
        p.len[h] += 1;
        p.ntok[i] += 1;
        if (p.label[i] != HKV_DENSE) p.nbuf[i] += 1;
      }
      if (tid == 0) *p.gcnt = 0;
    }
    __syncthreads();
  };
  const HeadLookup<FUSED> look{tab, p};
  TileIter cit;
  cit.h = tab.h0;
  cit.hs = tab.start[0];
  cit.hl = tab.vlen[0];
  cit.g = a;
  cit.b = b;

  // ---- producer state (warp 0, lane 0) ----------------------------------
  // A tile's old rows come from the arena; the query row (first tile of a
  // head here) and the new token's K/V (fused, last tile of a head) come from
  // this step's inputs, which may be written by the previous kernel.
  const bool producer = active && tid == 0;
  TileIter pit = cit;
  int issued = 0;
  auto issue_old = [&](Pending &pd) {  // expect + copy the arena rows, no arrival
    const int stage = issued % NS;
    const long long ge = pit.tile_end(TT);
    const int r0 = (int)(pit.g - pit.hs), r1 = (int)(ge - pit.hs);   // head-local rows
    const int real = FUSED ? pit.hl - 1 : pit.hl;                    // rows in the arena
    const int n_old = (r1 < real ? r1 : real) - r0;
    unsigned char *dk = stages + stage * S::kStageBytes;
    pd.h = pit.h;
    pd.slot_new = real - r0;
    pd.first = pit.g == pit.hs || pit.g == a;
    pd.has_new = FUSED && r1 == pit.hl;
    if (n_old > 0) {
      const uint32_t bytes = (uint32_t)n_old * RB;
      const long long row = look.off(pit.h) + r0;
      mbar_expect_tx(&full[stage], 2 * bytes);
      bulk_g2s(dk, static_cast<const unsigned char *>(p.K) + row * RB, bytes, &full[stage]);
      bulk_g2s(dk + TT * RB, static_cast<const unsigned char *>(p.V) + row * RB, bytes,
               &full[stage]);
    }
    pit.advance(TT, look);
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
    for (; n_pre < NS && !pit.done(); ++n_pre) issue_old(pre[n_pre]);

  if (p.prefetch) pdl_wait();  // the step's inputs are visible from here on
  if (tid == 0) HKV_TRACE(2);
  pdl_launch_dependents();
  if (early) grid_arrive();

  // Fused append of a head's new token (row, position, query) by the warp
  // that finishes the head; nothing in this launch reads them.
  auto append_row = [&](int h) {
    const int i = p.layer_base + h;
    const int jt = h - tab.h0;
    const bool in_tab = jt >= 0 && jt < tab.n;
    const int len = (in_tab ? tab.vlen[jt] : p.len[h] + 1) - 1;
    const int nt = in_tab ? tab.ntok[jt] : p.ntok[i];
    const long long row = look.off(h) + len;
    const uint4 *ks = reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(p.k_new) + (size_t)h * RB);
    const uint4 *vs = reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(p.v_new) + (size_t)h * RB);
    const uint4 *qs = reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(p.q) + (size_t)h * RB);
    uint4 *kd = reinterpret_cast<uint4 *>(static_cast<unsigned char *>(p.K) + row * RB);
    uint4 *vd = reinterpret_cast<uint4 *>(static_cast<unsigned char *>(p.V) + row * RB);
    uint4 *qd = reinterpret_cast<uint4 *>(static_cast<unsigned char *>(p.qbuf) +
                                          ((size_t)i * p.period + nt % p.period) * RB);
    for (int c = lane; c < RB / 16; c += 32) {
      kd[c] = ks[c];
      vd[c] = vs[c];
      qd[c] = qs[c];
    }
    if (lane == 0) p.pos[row] = p.n_cond + nt;
  };

  if (warp == 0) {
    // ---- producer ----------------------------------------------------------
    if (producer) {
#pragma unroll
      for (int j = 0; j < NS; ++j)
        if (j < n_pre) issue_extra(pre[j], j);
      while (!pit.done()) {
        const int stage = issued % NS;
        // the consumers are done with the tile that used this stage before
        if (s_abort || !mbar_wait(&empty[stage], (uint32_t)(issued / NS - 1) & 1u)) {
          s_abort = 1;
          set_err(p.err, HKV_ERR_TIMEOUT);
          break;
        }
        Pending pd;
        issue_old(pd);
        issue_extra(pd, stage);
      }
    }
  } else if (warp <= kCW) {
    // ---- consumers ---------------------------------------------------------
    const int ctid = tid - 32, cw = warp - 1;
    if (!FUSED && blockIdx.x == 0)  // empty heads (plain attention) are zeros
      for (int h = ctid; h < nheads; h += kCW * 32)
        if (p.len[h] == 0)
          for (int d = 0; d < D; ++d) p.out[(size_t)h * D + d] = 0.f;

    if (active) {
      const int grp = lane / LPR, col = lane % LPR;
      float q[EPL], acc[EPL];
      float m = -INFINITY, l = 0.f;
      int nseg = 0;
#pragma unroll
      for (int e = 0; e < EPL; ++e) acc[e] = 0.f;

      for (int tile = 0; !cit.done(); ++tile) {
        const int stage = tile % NS;
        if (!s_abort && !mbar_wait(&full[stage], (uint32_t)(tile / NS) & 1u)) {
          s_abort = 1;
          set_err(p.err, HKV_ERR_TIMEOUT);
        }
        if (tile == 0 && ctid == 0) HKV_TRACE(3);
        const long long ge = cit.tile_end(TT);
        const int n = (int)(ge - cit.g);
        const long long he = cit.hs + cit.hl;
        const unsigned char *Ks = stages + stage * S::kStageBytes;
        const unsigned char *Vs = Ks + TT * RB;
        if (cit.g == cit.hs || cit.g == a) {  // first tile of this head here
          Elem<T>::unpack(*reinterpret_cast<const uint4 *>(Vs + TT * RB + col * 16), q);
#pragma unroll
          for (int e = 0; e < EPL; ++e) {
            q[e] *= p.qscale;
            acc[e] = 0.f;
          }
          m = -INFINITY;
          l = 0.f;
        }

        float sc[S::kSteps];
#pragma unroll
        for (int st = 0; st < S::kSteps; ++st) {
          const int r = st * (kCW * RPW) + cw * RPW + grp;
          float dot = 0.f;
          if (r < n) {
            float kf[EPL];
            Elem<T>::unpack(*reinterpret_cast<const uint4 *>(Ks + r * RB + col * 16), kf);
#pragma unroll
            for (int e = 0; e < EPL; ++e) dot = fmaf(q[e], kf[e], dot);
          }
#pragma unroll
          for (int o = LPR / 2; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xFFFFFFFFu, dot, o);
          sc[st] = r < n ? dot : -INFINITY;
        }
        float mt = sc[0];
#pragma unroll
        for (int st = 1; st < S::kSteps; ++st) mt = fmaxf(mt, sc[st]);
        const float mn = fmaxf(m, mt);
        if (mn != -INFINITY) {
          const float corr = exp2f(m - mn);
          l *= corr;
#pragma unroll
          for (int e = 0; e < EPL; ++e) acc[e] *= corr;
#pragma unroll
          for (int st = 0; st < S::kSteps; ++st) {
            const int r = st * (kCW * RPW) + cw * RPW + grp;
            if (r < n) {
              const float pr = exp2f(sc[st] - mn);
              l += pr;
              float vf[EPL];
              Elem<T>::unpack(*reinterpret_cast<const uint4 *>(Vs + r * RB + col * 16), vf);
#pragma unroll
              for (int e = 0; e < EPL; ++e) acc[e] = fmaf(pr, vf[e], acc[e]);
            }
          }
          m = mn;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&empty[stage]);  // this warp is done with the stage
        if (ctid == 0 && ge == b) HKV_TRACE(4);

        if (ge == (b < he ? b : he)) {  // last tile of this head here: hand it over
#pragma unroll
          for (int o = LPR; o < 32; o <<= 1) {  // merge the row groups of the warp
            const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m, o);
            const float l2 = __shfl_xor_sync(0xFFFFFFFFu, l, o);
            const float mx = fmaxf(m, m2);
            const float s1 = m == -INFINITY ? 0.f : exp2f(m - mx);
            const float s2 = m2 == -INFINITY ? 0.f : exp2f(m2 - mx);
            l = l * s1 + l2 * s2;
#pragma unroll
            for (int e = 0; e < EPL; ++e) {
              const float a2 = __shfl_xor_sync(0xFFFFFFFFu, acc[e], o);
              acc[e] = acc[e] * s1 + a2 * s2;
            }
            m = mx;
          }
          // the epilogue is done with the previous segment's states
          if (nseg > 0 && !s_abort && !mbar_wait(&epi_free, (uint32_t)(nseg - 1) & 1u)) {
            s_abort = 1;
            set_err(p.err, HKV_ERR_TIMEOUT);
          }
          if (lane < LPR) {
#pragma unroll
            for (int e = 0; e < EPL; ++e) red_acc[cw][lane * EPL + e] = acc[e];
            if (lane == 0) {
              red_m[cw] = m;
              red_l[cw] = l;
            }
          }
          if (cw == 0 && lane == 0) {
            seg_h = cit.h;
            seg_hs = cit.hs;
            seg_he = he;
            seg_final = ge == b;
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&epi_full);
          ++nseg;
        }
        cit.advance(TT, look);
      }
      if (ctid == 0) HKV_TRACE(5);
      if (s_abort && ctid == 0)  // drain what may still be in flight (bounded)
        for (int s = 0; s < NS; ++s) {
          mbar_wait(&full[s], 0);
          mbar_wait(&full[s], 1);
        }
    }
  } else if (active) {
    // ---- epilogue: finish each head segment the consumers hand over --------
    constexpr int CPL = D / 32;  // output channels per lane
    for (int k = 0;; ++k) {
      if (!s_abort && !mbar_wait(&epi_full, (uint32_t)k & 1u)) {
        s_abort = 1;
        set_err(p.err, HKV_ERR_TIMEOUT);
      }
      if (s_abort) break;
      const int h = seg_h;
      const long long hs = seg_hs, he = seg_he;
      const int fin = seg_final;
      float mx = red_m[0];
#pragma unroll
      for (int w = 1; w < kCW; ++w) mx = fmaxf(mx, red_m[w]);
      float L = 0.f, A[CPL];
#pragma unroll
      for (int c = 0; c < CPL; ++c) A[c] = 0.f;
#pragma unroll
      for (int w = 0; w < kCW; ++w) {
        const float sw = red_m[w] == -INFINITY ? 0.f : exp2f(red_m[w] - mx);
        L += red_l[w] * sw;
#pragma unroll
        for (int c = 0; c < CPL; ++c) A[c] += red_acc[w][lane + 32 * c] * sw;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&epi_free);  // the consumers may reuse the slot
      if (hs >= a && he <= b) {  // the whole head is here
#pragma unroll
        for (int c = 0; c < CPL; ++c) p.out[(size_t)h * D + lane + 32 * c] = A[c] / L;
        if (FUSED) append_row(h);
      } else {
        float *pp = p.part + ((size_t)blockIdx.x * 2 + (hs <= a ? 0 : 1)) * (D + 2);
#pragma unroll
        for (int c = 0; c < CPL; ++c) pp[lane + 32 * c] = A[c];
        if (lane == 0) {
          pp[D] = mx;
          pp[D + 1] = L;
        }
        __syncwarp();
        const long long c0 = hs / chunk, c1 = (he - 1) / chunk;
        int last = 0;
        if (lane == 0) {
          __threadfence();
          last = atomicAdd(&p.cnt[h], 1) == (int)(c1 - c0);
        }
        last = __shfl_sync(0xFFFFFFFFu, last, 0);
        if (last) {  // the last CTA to arrive merges the pieces in CTA order
          __threadfence();
          float gm = -INFINITY, GL = 0.f, GA[CPL];
#pragma unroll
          for (int c = 0; c < CPL; ++c) GA[c] = 0.f;
          for (long long cc = c0; cc <= c1; ++cc) {
            const int slot = (cc == c0 && cc * chunk < hs) ? 1 : 0;
            const float *qq = p.part + ((size_t)cc * 2 + slot) * (D + 2);
            const float mc = __ldcg(qq + D), lc = __ldcg(qq + D + 1);
            const float mn2 = fmaxf(gm, mc);
            const float s0 = gm == -INFINITY ? 0.f : exp2f(gm - mn2);
            const float s1 = exp2f(mc - mn2);
            GL = GL * s0 + lc * s1;
#pragma unroll
            for (int c = 0; c < CPL; ++c) GA[c] = GA[c] * s0 + __ldcg(qq + lane + 32 * c) * s1;
            gm = mn2;
          }
#pragma unroll
          for (int c = 0; c < CPL; ++c) p.out[(size_t)h * D + lane + 32 * c] = GA[c] / GL;
          if (lane == 0) p.cnt[h] = 0;
          if (FUSED) append_row(h);
        }
      }
      if (fin) break;
    }
  }

  if (FUSED && !early) grid_arrive();  // the CTAs that read lengths late
  if (tid == 0) HKV_TRACE(6);
}

template <int D, typename T>
size_t smem_bytes() {
  return (size_t)AttnShape<D, T>::kNS * AttnShape<D, T>::kStageBytes;
}

template <int D, typename T, bool F>
cudaError_t prepare_t(int *ctas) {
  const size_t smem = smem_bytes<D, T>();
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<D, T, F>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas, attn_kernel<D, T, F>, kAttnThreads,
                                                       smem);
}

template <int D, typename T>
cudaError_t prepare_both(int *ctas) {
  int a = 0, b = 0;
  cudaError_t e = prepare_t<D, T, false>(&a);
  if (e != cudaSuccess) return e;
  e = prepare_t<D, T, true>(&b);
  *ctas = a < b ? a : b;
  if (*ctas > HKV_ATTN_MAX_CTAS_PER_SM) *ctas = HKV_ATTN_MAX_CTAS_PER_SM;
  return e;
}

template <int D, typename T>
cudaError_t launch_t(const AttnArgs &a, int grid, bool fused, cudaStream_t s) {
  static const bool pdl = getenv("HKV_NO_PDL") == nullptr;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kAttnThreads);
  cfg.dynamicSmemBytes = smem_bytes<D, T>();
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return fused ? cudaLaunchKernelEx(&cfg, attn_kernel<D, T, true>, a)
               : cudaLaunchKernelEx(&cfg, attn_kernel<D, T, false>, a);
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
  if (dtype == HKV_BF16) return D == 64 ? prepare_both<64, __nv_bfloat16>(ctas) : prepare_both<128, __nv_bfloat16>(ctas);
  return D == 64 ? prepare_both<64, float>(ctas) : prepare_both<128, float>(ctas);
}

cudaError_t launch_attention(const AttnArgs &a, int D, int dtype, int grid, bool fused,
                             cudaStream_t s) {
  if (dtype == HKV_BF16)
    return D == 64 ? launch_t<64, __nv_bfloat16>(a, grid, fused, s)
                   : launch_t<128, __nv_bfloat16>(a, grid, fused, s);
  return D == 64 ? launch_t<64, float>(a, grid, fused, s) : launch_t<128, float>(a, grid, fused, s);
}

}  // namespace hkv
