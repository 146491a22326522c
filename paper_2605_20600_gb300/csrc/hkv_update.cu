// Per-head cache maintenance of HeadKV, one CTA per head:
//  * evict / append_evict: the periodic head-aware update when a head's
//    buffer holds P tokens (Sec. 4: local heads drop their history, Eq. 3;
//    global heads trim it by Stratified Token Eviction, Eqs. 4-6), and for
//    append_evict the append of the new token after it (Sec. 3, KV Cache);
//  * repack: the first update at grouping, out of place from the dense
//    cache into the ragged one (Step 3);
//  * prefill / init_dense: the uncompressed cache of Step 1;
//  * identify: threshold-based attention accumulation (Step 2);
//  * budgets: per-head budgets and the arena layout (Sec. 5.1).
//
// The update works on token POSITIONS, not on storage order, so a segment
// may hold its live tokens in any order:
//  * conditioning tokens have positions < C; the recent window is the newest
//    w image tokens, positions >= C + ntok - w; everything else is history;
//  * Eq. 5's long-range subset is the floor(T * r_s) history tokens with the
//    smallest positions (a rank select on positions);
//  * scores q-bar . k in a fixed fp32 order, keys (order-preserving score
//    bits, position) unique and ascending in eviction priority, one 8-pass
//    MSD radix select finds the quota-th key of both subsets at once;
//  * in place, the holes below the new length are refilled with the
//    surviving rows above it: at most M rows move and no move depends on
//    another, instead of shifting every row after the first eviction.
#include <math.h>
#include <stdlib.h>

#include "hkv_device.cuh"
#include "hkv_kernels.h"

namespace hkv {
namespace {

constexpr int NT = kCacheThreads;
// update kernels resident per SM that the register budget allows (48
// registers a thread, no spills): a layer of many short heads (one CTA each)
// then runs in fewer waves; shared memory may allow fewer
constexpr int kUpdCtasPerSm = 5;

// Phase timestamps per head of the update for latency studies; compiled out
// by default.
#ifdef HKV_UPD_TRACE
__device__ unsigned long long *g_utrace = nullptr;  // [head of the layer][8], set by the tracer
#define HKV_UTRACE(slot)                                                   \
  do {                                                                     \
    if (g_utrace && threadIdx.x == 0)                                      \
      g_utrace[(size_t)blockIdx.x * 8 + (slot)] = globaltimer();           \
  } while (0)
#else
#define HKV_UTRACE(slot) \
  do {                   \
  } while (0)
#endif

__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

struct SegRef {
  const unsigned char *sk, *sv;  // source rows, row 0 = segment start
  const int32_t *spos;
  unsigned char *dk, *dv;        // destination rows
  int32_t *dpos;
  int len;                       // live source rows
  int dst_cap;                   // destination capacity (rows)
  bool in_place;
  uint32_t *err;                 // the cache's error word
};

struct UpdShared {
  unsigned long long prefix[2];
  int rem[2];
  int iscan[33];
  long long lscan[33];
  uint64_t ring_bar;  // completion of the bulk copy of the query ring
};

// Shared-memory work area of one update (dynamic).
struct UpdSmem {
  unsigned char *ring;       // [P][D] the buffered queries (<= 4 B each)
  unsigned long long *keys;  // [max_len]
  int *ps;                   // [max_len] positions of the source rows
  int *aux;                  // [max_len] class, then keep flag, then rank
  float *qbar;               // [D]
  int *hist;                 // [512]
  int stage_rows;            // rows a warp stages per pass of the score phase
};

// Rows a warp stages per pass of the score phase: 32, or fewer when every
// warp's share of the longest segment is smaller (short segments then leave
// room for more CTAs per SM).
__host__ __device__ constexpr int stage_rows(int max_len) {
  return max_len >= NT ? 32 : (max_len + NT / 32 - 1) / (NT / 32) < 1 ? 1 : (max_len + NT / 32 - 1) / (NT / 32);
}

// the query ring (P rows of es-byte elements); after q-bar it is the score
// stage: NT/32 warps x stage_rows rows of D * es + 16 bytes
__host__ __device__ constexpr size_t ring_bytes(int P, int D, int es, int max_len) {
  return (size_t)P * D * es > (size_t)(NT / 32) * stage_rows(max_len) * (D * es + 16)
             ? (size_t)P * D * es
             : (size_t)(NT / 32) * stage_rows(max_len) * (D * es + 16);
}

__device__ __forceinline__ UpdSmem carve(unsigned char *dyn, int max_len, int D, int P, int es) {
  UpdSmem u;
  u.ring = dyn;
  u.stage_rows = stage_rows(max_len);
  u.keys = reinterpret_cast<unsigned long long *>(dyn + ring_bytes(P, D, es, max_len));
  u.ps = reinterpret_cast<int *>(u.keys + max_len);
  u.aux = u.ps + max_len;
  u.qbar = reinterpret_cast<float *>(u.aux + max_len);
  u.hist = reinterpret_cast<int *>(u.qbar + D);
  return u;
}

// The k0-th smallest key among rows of class 0 and the k1-th among rows of
// class 1 (1-based; 0 = not needed; other classes ignored), by MSD radix
// select on bytes from `top_shift` down. Keys are unique within a class, so
// each result bounds exactly k keys of its class from above.
__device__ void radix_select2(const unsigned long long *keys, const int *cls, int n, int k0,
                              int k1, int top_shift, int *hist, UpdShared &sh) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) {
    sh.prefix[0] = sh.prefix[1] = 0ull;
    sh.rem[0] = k0;
    sh.rem[1] = k1;
  }
  __syncthreads();
  for (int shift = top_shift; shift >= 0; shift -= 8) {
    for (int i = tid; i < 512; i += NT) hist[i] = 0;
    __syncthreads();
    const unsigned long long hi = shift >= 56 ? 0ull : (~0ull << (shift + 8));
    const unsigned long long p0 = sh.prefix[0], p1 = sh.prefix[1];
    const int r0 = sh.rem[0], r1 = sh.rem[1];
    for (int j = tid; j < n; j += NT) {
      const int s = cls[j];
      if (s != 0 && s != 1) continue;
      const unsigned long long key = keys[j];
      if ((s ? r1 : r0) > 0 && (key & hi) == (s ? p1 : p0))
        atomicAdd(&hist[s * 256 + (int)((key >> shift) & 255ull)], 1);
    }
    __syncthreads();
    if (warp < 2) {
      const int s = warp;
      const int target = sh.rem[s];
      if (target > 0) {  // warp-uniform
        int c[8], sum = 0;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          c[e] = hist[s * 256 + lane * 8 + e];
          sum += c[e];
        }
        const int incl = warp_incl_scan(sum);
        const int excl = incl - sum;
        if (excl < target && target <= incl) {
          int run = excl, digit = -1, rem = 0, in_bin = 0;
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            if (digit < 0 && run + c[e] >= target) {
              digit = lane * 8 + e;
              rem = target - run;
              in_bin = c[e];
            }
            run += c[e];
          }
          sh.prefix[s] |= (unsigned long long)digit << shift;
          if (rem == in_bin) {
            // every key of this bin is among the k: the bin's upper end
            // bounds exactly k keys (keys are unique), no further digit
            sh.prefix[s] |= shift > 0 ? (1ull << shift) - 1ull : 0ull;
            sh.rem[s] = 0;
          } else {
            sh.rem[s] = rem;
          }
        }
      }
    }
    __syncthreads();
    if (sh.rem[0] == 0 && sh.rem[1] == 0) break;
  }
}

__device__ __forceinline__ int block_sum(int x, UpdShared &sh) {
  int tot;
  block_excl_scan<int>(x, sh.iscan, &tot);
  return tot;
}

// Decides which rows of a segment the update evicts (Eqs. 2-6). On return
// u.aux[r] is 1 for a kept row and 0 for an evicted one (r < len), u.ps
// holds the rows' positions, and the number of evicted rows is returned.
// Block-uniform.
template <int D, typename T>
__device__ int select_evictions(const SegRef &sg, int label, const MethodArgs &m,
                                const unsigned char *qring, int ntok, const UpdSmem &u,
                                UpdShared &sh) {
  constexpr int RB = D * (int)sizeof(T);
  constexpr int EPL = Elem<T>::kPerPiece;
  constexpr int LPR = RB / 16;
  const int tid = threadIdx.x;
  const int C = m.C;
  const int recent_from = C + (ntok > m.w ? ntok - m.w : 0);   // newest w image tokens
  int nh = 0;
  for (int r = tid; r < sg.len; r += NT) {
    const int ps = sg.spos[r];
    u.ps[r] = ps;
    const bool hist = ps >= C && ps < recent_from;
    u.aux[r] = hist ? 0 : -1;   // class: history (0) or always kept (-1)
    nh += hist ? 1 : 0;
  }
  const int NH = block_sum(nh, sh);  // history candidates (Eq. 2)
  HKV_UTRACE(1);
  // the head's history budget, B_g - w with the paper's budgets, from the
  // capacity its segment was given (C + budget + P)
  const int hist_budget = sg.dst_cap - C - m.P - m.w > 0 ? sg.dst_cap - C - m.P - m.w : 0;
  int M = 0;
  if (label == HKV_LOCAL) M = NH;    // Eq. 3: no history
  else if (NH > hist_budget) M = NH - hist_budget;

  if (label == HKV_GLOBAL && M > 0) {
    // Eq. 5: the floor(NH r_s) oldest history tokens are long-range (or,
    // in the grid-distance variant, the farthest from the newest image
    // token, equal distances older first)
    const int n_long = (int)floor((double)NH * m.r_s);
    if (n_long > 0 && n_long < NH && m.grid2d) {
      const int ref = ntok - 1;
      for (int r = tid; r < sg.len; r += NT) {
        const int i = u.ps[r] - C;
        const long long dr = i / m.row_len - ref / m.row_len, dc = i % m.row_len - ref % m.row_len;
        const unsigned long long far = 0x7FFFFFFFull - (unsigned long long)(dr * dr + dc * dc);
        u.keys[r] = (far << 32) | (uint32_t)u.ps[r];
      }
      radix_select2(u.keys, u.aux, sg.len, n_long, 0, 56, u.hist, sh);
      const unsigned long long k_long = sh.prefix[0];
      for (int r = tid; r < sg.len; r += NT)
        if (u.aux[r] == 0) u.aux[r] = u.keys[r] <= k_long ? 0 : 1;
    } else if (n_long > 0 && n_long < NH) {
      for (int r = tid; r < sg.len; r += NT) u.keys[r] = (unsigned long long)(uint32_t)u.ps[r];
      const int maxp = C + ntok;  // positions are below it: start at its top byte
      const int top = maxp < (1 << 8) ? 0 : maxp < (1 << 16) ? 8 : maxp < (1 << 24) ? 16 : 24;
      radix_select2(u.keys, u.aux, sg.len, n_long, 0, top, u.hist, sh);
      const int p_long = (int)sh.prefix[0];
      for (int r = tid; r < sg.len; r += NT)
        if (u.aux[r] == 0) u.aux[r] = u.ps[r] <= p_long ? 0 : 1;
    } else {
      for (int r = tid; r < sg.len; r += NT)
        if (u.aux[r] == 0) u.aux[r] = n_long == NH ? 0 : 1;
    }
    HKV_UTRACE(2);
    // Eq. 6 scores: q-bar = the P buffered queries, oldest first. The ring
    // comes in with one bulk copy; the sums keep their order.
    const int P = m.P;
    if (tid == 0) {
      mbar_init(&sh.ring_bar, 1);
      fence_barrier_init();
    }
    __syncthreads();
    if (tid == 0) {
      const uint32_t bytes = (uint32_t)P * RB;
      mbar_arrive_expect_tx(&sh.ring_bar, bytes);
      bulk_g2s(u.ring, qring, bytes, &sh.ring_bar);
    }
    if (!mbar_wait(&sh.ring_bar, 0) && tid == 0) set_err(sg.err, HKV_ERR_TIMEOUT);
    for (int d = tid; d < D; d += NT) {
      float acc = 0.f;
      for (int pp = 0; pp < P; ++pp) {
        int slot = (ntok - P + pp) % P;
        if (slot < 0) slot += P;
        acc = __fadd_rn(acc, Elem<T>::load1(u.ring, (size_t)slot * D + d));
      }
      u.qbar[d] = acc;
    }
    __syncthreads();
    HKV_UTRACE(3);
    // Each warp stages 32 rows at a time in the (now free) ring area with
    // coalesced 16-byte async copies, at a row stride of LPR + 1 pieces so
    // that lane l reading row l, piece j, hits distinct banks; then lane l
    // sums its row in the fixed order.
    constexpr int RS = LPR + 1;  // row stride in 16-byte pieces
    const int warp = tid >> 5, lane = tid & 31;
    const int SR = u.stage_rows;
    unsigned char *stage = u.ring + (size_t)warp * SR * RS * 16;
    for (int base = warp * SR; base < sg.len; base += (NT / 32) * SR) {
      const int nrows = sg.len - base < SR ? sg.len - base : SR;
      for (int w = lane; w < nrows * LPR; w += 32) {
        const int rr = w / LPR, pc = w % LPR;
        cp_async16(stage + (rr * RS + pc) * 16, sg.sk + (size_t)(base + rr) * RB + pc * 16);
      }
      cp_async_wait_all();
      __syncwarp();
      const int r = base + lane;
      if (lane < nrows && u.aux[r] >= 0) {
        const unsigned char *krow = stage + lane * RS * 16;
        float s = 0.f;
#pragma unroll 4
        for (int pc = 0; pc < LPR; ++pc) {
          float kf[EPL];
          Elem<T>::unpack(*reinterpret_cast<const uint4 *>(krow + pc * 16), kf);
#pragma unroll
          for (int e = 0; e < EPL; ++e) s = __fadd_rn(s, __fmul_rn(u.qbar[pc * EPL + e], kf[e]));
        }
        s = __fadd_rn(s, 0.f);  // -0 reads as +0
        uint32_t bits = __float_as_uint(s);
        bits = (bits & 0x80000000u) ? ~bits : (bits | 0x80000000u);  // order-preserving
        u.keys[r] = ((unsigned long long)bits << 32) | (uint32_t)u.ps[r];
      }
      __syncwarp();  // the stage is rewritten next round
    }
    __syncthreads();
    HKV_UTRACE(4);
    // M/2 from each subset; a short subset hands its excess to the other
    int m_long = M / 2, m_near = M - M / 2;
    if (m_long > n_long) {
      m_near += m_long - n_long;
      m_long = n_long;
    }
    if (m_near > NH - n_long) {
      m_long += m_near - (NH - n_long);
      m_near = NH - n_long;
    }
    radix_select2(u.keys, u.aux, sg.len, m_long, m_near, 56, u.hist, sh);
    const unsigned long long thr0 = sh.prefix[0], thr1 = sh.prefix[1];
    for (int r = tid; r < sg.len; r += NT) {
      const int c = u.aux[r];
      const bool ev = c == 0 ? (m_long > 0 && u.keys[r] <= thr0)
                             : c == 1 ? (m_near > 0 && u.keys[r] <= thr1) : false;
      u.aux[r] = ev ? 0 : 1;
    }
    HKV_UTRACE(5);
  } else {
    for (int r = tid; r < sg.len; r += NT) u.aux[r] = (u.aux[r] == 0 && M > 0) ? 0 : 1;
  }
  __syncthreads();
  return M;
}

template <int D, typename T>
__device__ __forceinline__ void copy_piece(unsigned char *dk, unsigned char *dv,
                                           const unsigned char *sk, const unsigned char *sv,
                                           int piece) {
  *reinterpret_cast<uint4 *>(dk + piece * 16) =
      __ldcg(reinterpret_cast<const uint4 *>(sk + piece * 16));
  *reinterpret_cast<uint4 *>(dv + piece * 16) =
      __ldcg(reinterpret_cast<const uint4 *>(sv + piece * 16));
}

// In place: the new length is len - M; every evicted row below it takes a
// surviving row from above it (the i-th hole the i-th survivor). Sources
// are all >= new_len and destinations < new_len, so the moves are
// independent. Each thread ranks a contiguous run of rows (one block scan
// for holes and fills together), and each copy batch issues all of its
// loads before its stores. Returns the new length.
template <int D, typename T>
__device__ int fill_holes(const SegRef &sg, int M, const UpdSmem &u, UpdShared &sh) {
  constexpr int RB = D * (int)sizeof(T);
  constexpr int LPR = RB / 16;
  constexpr int B = 4;  // pieces per thread in flight
  const int tid = threadIdx.x;
  const int len = sg.len, new_len = len - M;
  if (M == 0) return len;
  // the keys area is free now and holds the two index lists
  int *hole = reinterpret_cast<int *>(u.keys);  // [M]
  int *fill = hole + M;                          // [M]
  const int per = (len + NT - 1) / NT;
  const int r0 = tid * per < len ? tid * per : len;
  const int r1 = r0 + per < len ? r0 + per : len;
  long long nh = 0, nf = 0;
  for (int r = r0; r < r1; ++r) {
    const int keep = u.aux[r];
    nh += (r < new_len && !keep) ? 1 : 0;
    nf += (r >= new_len && keep) ? 1 : 0;
  }
  long long tot;
  const long long ex = block_excl_scan<long long>((nh << 32) | nf, sh.lscan, &tot);
  int hp = (int)(ex >> 32), fp = (int)(ex & 0xFFFFFFFFll);
  for (int r = r0; r < r1; ++r) {
    const int keep = u.aux[r];
    if (r < new_len && !keep) hole[hp++] = r;
    if (r >= new_len && keep) fill[fp++] = r;
  }
  __syncthreads();
  const int k = (int)(tot >> 32);  // = M: holes and fills pair up
  const int total = k * LPR;
  for (int w0 = 0; w0 < total; w0 += NT * B) {
    uint4 kb[B], vb[B];
#pragma unroll
    for (int j = 0; j < B; ++j) {
      const int w = w0 + j * NT + tid;
      if (w < total) {
        const size_t src = (size_t)fill[w / LPR] * RB + (w % LPR) * 16;
        kb[j] = __ldcg(reinterpret_cast<const uint4 *>(sg.sk + src));
        vb[j] = __ldcg(reinterpret_cast<const uint4 *>(sg.sv + src));
      }
    }
#pragma unroll
    for (int j = 0; j < B; ++j) {
      const int w = w0 + j * NT + tid;
      if (w < total) {
        const size_t dst = (size_t)hole[w / LPR] * RB + (w % LPR) * 16;
        *reinterpret_cast<uint4 *>(sg.dk + dst) = kb[j];
        *reinterpret_cast<uint4 *>(sg.dv + dst) = vb[j];
      }
    }
  }
  for (int j = tid; j < k; j += NT) sg.dpos[hole[j]] = u.ps[fill[j]];
  __syncthreads();
  return new_len;
}

// Out of place, keeping the source order: survivors are packed by a prefix
// sum of the keep flags. Returns the new length.
template <int D, typename T>
__device__ int copy_kept(const SegRef &sg, const UpdSmem &u, UpdShared &sh) {
  constexpr int RB = D * (int)sizeof(T);
  constexpr int LPR = RB / 16;
  const int tid = threadIdx.x;
  int run = 0;
  for (int base = 0; base < sg.len; base += NT) {
    const int r = base + tid;
    const int keep = r < sg.len ? u.aux[r] : 0;
    int tot;
    const int ex = block_excl_scan<int>(keep, sh.iscan, &tot);
    if (r < sg.len) u.aux[r] = keep ? run + ex : -1;
    run += tot;
  }
  __syncthreads();
  for (int w = tid; w < sg.len * LPR; w += NT) {
    const int r = w / LPR, pc = w % LPR;
    const int d = u.aux[r];
    if (d >= 0)
      copy_piece<D, T>(sg.dk + (size_t)d * RB, sg.dv + (size_t)d * RB, sg.sk + (size_t)r * RB,
                       sg.sv + (size_t)r * RB, pc);
  }
  for (int r = tid; r < sg.len; r += NT)
    if (u.aux[r] >= 0) sg.dpos[u.aux[r]] = u.ps[r];
  __syncthreads();
  return run;
}

// The update of one head in place (local: window slide; global: STE).
template <int D, typename T>
__device__ int update_in_place(const SegRef &sg, int label, const MethodArgs &m,
                               const unsigned char *qring, int ntok, const UpdSmem &u,
                               UpdShared &sh) {
  const int M = select_evictions<D, T>(sg, label, m, qring, ntok, u, sh);
  return fill_holes<D, T>(sg, M, u, sh);
}

template <int D, typename T>
__global__ void __launch_bounds__(NT, kUpdCtasPerSm)
    evict_kernel(const CacheArgs c, const MethodArgs m, int layer_base, int max_len) {
  constexpr int RB = D * (int)sizeof(T);
  extern __shared__ __align__(16) unsigned char dyn[];
  __shared__ UpdShared sh;
  // no early launch of the next kernel: a decode step that prefetches this
  // layer's cache before its own wait must start after the update is done
  pdl_wait();
  const int tid = threadIdx.x, i = layer_base + blockIdx.x;
  const uint8_t lab = c.label[i];
  const int nbuf = c.nbuf[i];
  if (lab == HKV_DENSE || nbuf < m.P) return;  // not due
  const int len = c.len[i], cp = c.cap[i];
  const long long off = c.off[i];
  if (off < 0 || cp < 0 || off + cp > c.arena_tokens || len < 0 || len > cp) {
    if (tid == 0) set_err(c.err, HKV_ERR_BOUNDS);
    return;
  }
  if (len > max_len) {
    if (tid == 0) set_err(c.err, HKV_ERR_CAPACITY);
    return;
  }
  unsigned char *K = static_cast<unsigned char *>(c.K) + off * RB;
  unsigned char *V = static_cast<unsigned char *>(c.V) + off * RB;
  int32_t *pos = c.pos + off;
  const unsigned char *qring = static_cast<const unsigned char *>(c.qbuf) + (size_t)i * m.P * RB;
  SegRef sg{K, V, pos, K, V, pos, len, cp, true, c.err};
  HKV_UTRACE(0);
  const int nl =
      update_in_place<D, T>(sg, lab, m, qring, c.ntok[i], carve(dyn, max_len, D, m.P, (int)sizeof(T)), sh);
  HKV_UTRACE(6);
  if (tid == 0) {
    c.len[i] = nl;
    c.nbuf[i] = 0;
  }
}

template <int D, typename T>
__global__ void __launch_bounds__(NT, kUpdCtasPerSm)
    append_evict_kernel(const CacheArgs c, const MethodArgs m, int layer_base, const void *q,
                        const void *k, const void *v, int max_len) {
  constexpr int RB = D * (int)sizeof(T);
  extern __shared__ __align__(16) unsigned char dyn[];
  __shared__ UpdShared sh;
  pdl_wait();
  pdl_launch_dependents();
  const int tid = threadIdx.x, hl = blockIdx.x, i = layer_base + hl;
  int len = c.len[i];
  const int cp = c.cap[i];
  const long long off = c.off[i];
  const uint8_t lab = c.label[i];
  const int ntok = c.ntok[i];
  int nbuf = c.nbuf[i];
  if (off < 0 || cp < 0 || off + cp > c.arena_tokens || len < 0 || len > cp) {
    if (tid == 0) set_err(c.err, HKV_ERR_BOUNDS);
    return;
  }
  unsigned char *K = static_cast<unsigned char *>(c.K) + off * RB;
  unsigned char *V = static_cast<unsigned char *>(c.V) + off * RB;
  int32_t *pos = c.pos + off;
  const unsigned char *qring = static_cast<const unsigned char *>(c.qbuf) + (size_t)i * m.P * RB;

  if (lab != HKV_DENSE && nbuf >= m.P) {  // buffer full: head-aware update
    if (len > max_len) {
      if (tid == 0) set_err(c.err, HKV_ERR_CAPACITY);
      return;
    }
    SegRef sg{K, V, pos, K, V, pos, len, cp, true, c.err};
    len = update_in_place<D, T>(sg, lab, m, qring, ntok, carve(dyn, max_len, D, m.P, (int)sizeof(T)), sh);
    nbuf = 0;
  }
  if (len >= cp) {
    if (tid == 0) {
      set_err(c.err, HKV_ERR_CAPACITY);
      c.len[i] = len;
      c.nbuf[i] = nbuf;
    }
    return;
  }
  // append the new token (K <- [K, k_t], V <- [V, v_t]) and its query
  const size_t row = (size_t)len;
  unsigned char *qdst = static_cast<unsigned char *>(c.qbuf) + ((size_t)i * m.P + ntok % m.P) * RB;
  for (int pc = tid; pc < RB / 16; pc += NT) {
    const size_t src = (size_t)hl * RB + pc * 16;
    *reinterpret_cast<uint4 *>(K + row * RB + pc * 16) =
        *reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(k) + src);
    *reinterpret_cast<uint4 *>(V + row * RB + pc * 16) =
        *reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(v) + src);
    *reinterpret_cast<uint4 *>(qdst + pc * 16) =
        *reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(q) + src);
  }
  if (tid == 0) {
    pos[row] = m.C + ntok;
    c.len[i] = len + 1;
    c.ntok[i] = ntok + 1;
    if (lab != HKV_DENSE) c.nbuf[i] = nbuf + 1;
  }
}

template <int D, typename T>
__global__ void __launch_bounds__(NT, kUpdCtasPerSm)
    repack_kernel(const CacheArgs dn, const CacheArgs rg, const MethodArgs m, int layer_base,
                  int max_len) {
  constexpr int RB = D * (int)sizeof(T);
  extern __shared__ __align__(16) unsigned char dyn[];
  __shared__ UpdShared sh;
  pdl_wait();
  pdl_launch_dependents();
  const int tid = threadIdx.x, i = layer_base + blockIdx.x;
  const int slen = dn.len[i];
  const long long soff = dn.off[i];
  const long long doff = rg.off[i];
  const int dcap = rg.cap[i];
  const uint8_t lab = rg.label[i];
  if (lab != HKV_LOCAL && lab != HKV_GLOBAL) {
    if (tid == 0) set_err(rg.err, HKV_ERR_STATE);
    return;
  }
  if (soff < 0 || slen < 0 || soff + slen > dn.arena_tokens || doff < 0 || dcap < 0 ||
      doff + dcap > rg.arena_tokens) {
    if (tid == 0) set_err(rg.err, HKV_ERR_BOUNDS);
    return;
  }
  if (slen > max_len) {
    if (tid == 0) set_err(rg.err, HKV_ERR_CAPACITY);
    return;
  }
  SegRef sg{static_cast<const unsigned char *>(dn.K) + soff * RB,
            static_cast<const unsigned char *>(dn.V) + soff * RB,
            dn.pos + soff,
            static_cast<unsigned char *>(rg.K) + doff * RB,
            static_cast<unsigned char *>(rg.V) + doff * RB,
            rg.pos + doff,
            slen,
            dcap,
            false,
            rg.err};
  const unsigned char *qring = static_cast<const unsigned char *>(dn.qbuf) + (size_t)i * m.P * RB;
  const UpdSmem u = carve(dyn, max_len, D, m.P, (int)sizeof(T));
  const int M = select_evictions<D, T>(sg, lab, m, qring, dn.ntok[i], u, sh);
  if (slen - M > dcap) {
    if (tid == 0) set_err(rg.err, HKV_ERR_CAPACITY);
    return;
  }
  const int nl = copy_kept<D, T>(sg, u, sh);
  if (tid == 0) {
    rg.len[i] = nl;
    rg.nbuf[i] = 0;
    rg.ntok[i] = dn.ntok[i];
  }
}

template <int D, typename T>
__global__ void prefill_kernel(const CacheArgs c, int layer_base, int C, const void *kc,
                               const void *vc) {
  constexpr int RB = D * (int)sizeof(T);
  pdl_wait();
  pdl_launch_dependents();
  const int hl = blockIdx.x, i = layer_base + hl, tid = threadIdx.x;
  const long long off = c.off[i];
  const int cp = c.cap[i];
  if (c.label[i] != HKV_DENSE || c.len[i] != 0) {
    if (tid == 0) set_err(c.err, HKV_ERR_STATE);
    return;
  }
  if (off < 0 || cp < C || off + cp > c.arena_tokens) {
    if (tid == 0) set_err(c.err, cp < C ? HKV_ERR_CAPACITY : HKV_ERR_BOUNDS);
    return;
  }
  const int pieces = C * (RB / 16);
  for (int pc = tid; pc < pieces; pc += blockDim.x) {
    const size_t src = (size_t)hl * C * RB + (size_t)pc * 16;
    const size_t dst = (size_t)off * RB + (size_t)pc * 16;
    *reinterpret_cast<uint4 *>(static_cast<unsigned char *>(c.K) + dst) =
        *reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(kc) + src);
    *reinterpret_cast<uint4 *>(static_cast<unsigned char *>(c.V) + dst) =
        *reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(vc) + src);
  }
  for (int j = tid; j < C; j += blockDim.x) c.pos[off + j] = j;
  if (tid == 0) {
    c.len[i] = C;
    c.nbuf[i] = 0;
    c.ntok[i] = 0;
  }
}

__global__ void init_dense_kernel(const CacheArgs c, int n, int seg) {
  pdl_wait();
  pdl_launch_dependents();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    const_cast<int64_t *>(c.off)[i] = (int64_t)i * seg;
    const_cast<int32_t *>(c.cap)[i] = seg;
    c.len[i] = 0;
    c.nbuf[i] = 0;
    c.ntok[i] = 0;
    const_cast<uint8_t *>(c.label)[i] = HKV_DENSE;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) *c.err = 0u;
}

// Row steps of the identification kernels' logit loops whose key loads are
// issued before the first is used (one step at a time costs a memory round
// trip per step). Measured on a GB300 (one call per layer): dense segments
// of 628 tokens or more go faster with 8 (single query; 26 -> 14 us per
// layer at 628) or 4 (multi-query: -19 % at 628, -35 % at 2128 tokens) than
// with one; segments of 101-164 tokens go best with 2, where more loads in
// flight cost registers and resident CTAs.
constexpr int kIdLongSegment = 512;
__host__ __device__ constexpr int id_rows_in_flight(int max_len, bool multi) {
  return max_len >= kIdLongSegment ? (multi ? 4 : 8) : 2;
}

// Shared memory of the identification kernels beyond their weights: in the
// grid-distance variant, the order keys ([max_len] 64-bit, 8-byte aligned
// after `floats` floats) and the count order ([max_len] int).
__host__ __device__ constexpr size_t id_order_offset(size_t floats) {
  return (floats * 4 + 7) / 8 * 8;
}
__host__ __device__ constexpr size_t id_smem(size_t floats, int max_len, bool grid2d) {
  return grid2d ? id_order_offset(floats) + (size_t)max_len * 12 : floats * 4;
}

// The count order of the grid-distance variant of Step 2: perm[j] = the row
// of the j-th token counted. Image tokens by squared grid distance from image
// token ref, nearest first, equal distances newer first; then the
// conditioning tokens, newest first. Keys are unique (positions are); each
// row's rank is the number of smaller keys (len^2 / NT comparisons per
// thread, once per head and generation). Block-uniform.
__device__ void grid_count_order(const int32_t *pos, int len, int C, int row_len, int ref,
                                 unsigned long long *keys, int *perm) {
  for (int r = threadIdx.x; r < len; r += blockDim.x) {
    const int p = pos[r];
    const unsigned long long newer = 0xFFFFFFFFull - (uint32_t)p;
    unsigned long long key = (1ull << 63) | newer;  // conditioning: after every image token
    if (p >= C) {
      const int i = p - C;
      const long long dr = i / row_len - ref / row_len, dc = i % row_len - ref % row_len;
      key = ((unsigned long long)(dr * dr + dc * dc) << 32) | newer;
    }
    keys[r] = key;
    perm[r] = r;  // a valid row for every slot even if positions repeat
  }
  __syncthreads();
  for (int r = threadIdx.x; r < len; r += blockDim.x) {
    const unsigned long long k = keys[r];
    int rank = 0;
    for (int j = 0; j < len; ++j) rank += keys[j] < k ? 1 : 0;
    perm[rank] = r;
  }
  __syncthreads();
}

// Step 2: attention of the current query over the key cache, accumulated
// backward from the newest token until tau (or outward on the grid in the
// grid-distance variant); local iff fewer than w_loc tokens were needed.
// The dense cache holds its tokens in position order.
template <int D, typename T, int U>
__global__ void __launch_bounds__(NT)
    identify_kernel(const CacheArgs c, const MethodArgs m, int layer_base, const void *q,
                    uint8_t *label_out, int32_t *nh_out, float qscale, int max_len) {
  constexpr int RB = D * (int)sizeof(T);
  constexpr int EPL = Elem<T>::kPerPiece;
  constexpr int LPR = RB / 16;
  constexpr int RPW = 32 / LPR;
  constexpr int NW = NT / 32;
  extern __shared__ float e[];
  __shared__ float red[NW];
  __shared__ float s_bcast;
  __shared__ float fscan[33];
  __shared__ int s_nh;
  pdl_wait();
  pdl_launch_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int hl = blockIdx.x, i = layer_base + hl;
  const int len = c.len[i];
  const long long off = c.off[i];
  if (c.label[i] != HKV_DENSE) {  // only the uncompressed cache is in order
    if (tid == 0) set_err(c.err, HKV_ERR_STATE);
    return;
  }
  if (off < 0 || len <= 0 || off + len > c.arena_tokens) {
    if (tid == 0) set_err(c.err, HKV_ERR_BOUNDS);
    return;
  }
  if (len > max_len) {  // the attention row must fit in shared memory
    if (tid == 0) set_err(c.err, HKV_ERR_CAPACITY);
    return;
  }
  const int grp = lane / LPR, col = lane % LPR;
  float qf[EPL];
  Elem<T>::unpack(*reinterpret_cast<const uint4 *>(static_cast<const unsigned char *>(q) +
                                                   (size_t)hl * RB + col * 16),
                  qf);
#pragma unroll
  for (int x = 0; x < EPL; ++x) qf[x] *= qscale;
  const unsigned char *K = static_cast<const unsigned char *>(c.K) + off * RB;
  // logits (log2 units); U row steps load before any is used
  for (int r0 = warp * RPW; r0 < len; r0 += U * NW * RPW) {
    uint4 kr[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int r = r0 + u * NW * RPW + grp;
      kr[u] = r < len ? *reinterpret_cast<const uint4 *>(K + (size_t)r * RB + col * 16)
                      : make_uint4(0u, 0u, 0u, 0u);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int r = r0 + u * NW * RPW + grp;
      float kf[EPL];
      Elem<T>::unpack(kr[u], kf);
      float dot = 0.f;
#pragma unroll
      for (int x = 0; x < EPL; ++x) dot = fmaf(qf[x], kf[x], dot);
#pragma unroll
      for (int o = LPR / 2; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xFFFFFFFFu, dot, o);
      if (r < len && col == 0) e[r] = dot;
    }
  }
  __syncthreads();
  float mx = -INFINITY;
  for (int r = tid; r < len; r += NT) mx = fmaxf(mx, e[r]);
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, o));
  if (lane == 0) red[warp] = mx;
  __syncthreads();
  if (tid == 0) {
    float v = red[0];
    for (int w = 1; w < NW; ++w) v = fmaxf(v, red[w]);
    s_bcast = v;
  }
  __syncthreads();
  mx = s_bcast;
  float sum = 0.f;
  for (int r = tid; r < len; r += NT) {
    const float x = exp2f(e[r] - mx);
    e[r] = x;
    sum += x;
  }
#pragma unroll
  for (int o = 16; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, o);
  __syncthreads();
  if (lane == 0) red[warp] = sum;
  __syncthreads();
  if (tid == 0) {
    float v = 0.f;
    for (int w = 0; w < NW; ++w) v += red[w];
    s_bcast = v * m.tau;
    s_nh = len;
  }
  __syncthreads();
  const float thr = s_bcast;
  int *perm = nullptr;
  if (m.grid2d) {
    unsigned char *base = reinterpret_cast<unsigned char *>(e) + id_order_offset(max_len);
    perm = reinterpret_cast<int *>(base + (size_t)max_len * 8);
    grid_count_order(c.pos + off, len, m.C, m.row_len, c.ntok[i] - 1,
                     reinterpret_cast<unsigned long long *>(base), perm);
  }
  float running = 0.f;  // cumulative mass from the newest token
  for (int base = 0; base < len; base += NT) {
    const int jb = base + tid;  // jb-th token counted (0 = current)
    const float x = jb < len ? e[perm ? perm[jb] : len - 1 - jb] : 0.f;
    float tot;
    const float cum = running + block_excl_scan<float>(x, fscan, &tot) + x;
    if (jb < len && cum >= thr) atomicMin(&s_nh, jb + 1);
    running += tot;
  }
  __syncthreads();
  if (tid == 0) {
    label_out[i] = s_nh < m.w_loc ? HKV_LOCAL : HKV_GLOBAL;
    if (nh_out) nh_out[i] = s_nh;
  }
}

// Block-wide max (MAX) or sum of N floats per thread, returned to every
// thread in place; red holds N values per warp, bc the N results.
// Consecutive calls are safe: each reads its operands before the next call
// writes them.
template <bool MAX, int N>
__device__ __forceinline__ void block_all(float (&v)[N], float *red, float *bc) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int b = 0; b < N; ++b) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      const float u = __shfl_xor_sync(0xFFFFFFFFu, v[b], o);
      v[b] = MAX ? fmaxf(v[b], u) : v[b] + u;
    }
    if (lane == 0) red[b * nw + warp] = v[b];
  }
  __syncthreads();
  if (threadIdx.x < N) {
    const int b = threadIdx.x;
    float a = red[b * nw];
    for (int w = 1; w < nw; ++w) a = MAX ? fmaxf(a, red[b * nw + w]) : a + red[b * nw + w];
    bc[b] = a;
  }
  __syncthreads();
#pragma unroll
  for (int b = 0; b < N; ++b) v[b] = bc[b];
}

// queries of the multi-query identification handled per pass over the keys:
// 8 for rings of at least kIdQB8From queries, else 4 (measured on a GB300:
// 8 is 17 % faster on 65-query rings over 628 keys, 4 is 26-33 % faster on
// 24-query rings over 101-164 keys, where the fewer registers of 4 give
// more CTAs per SM)
#ifndef HKV_ID_QB8_FROM
#define HKV_ID_QB8_FROM 48
#endif
constexpr int kIdQB8From = HKV_ID_QB8_FROM;
__host__ __device__ constexpr int id_qb(int P) { return P >= kIdQB8From ? 8 : 4; }

// Multi-query variant of Step 2 (not in the paper): the newest Pe = min(P,
// ntok) queries of the ring each attend over the keys that existed at their
// own step (the p-th oldest of them over the oldest len - (Pe - 1 - p)
// keys), their normalised attention rows are averaged, and the average is
// accumulated backward from the newest token until tau, as in
// identify_kernel. One CTA per head; each pass over the keys serves QB
// queries (every key row loaded once per pass, dotted with all of them).
template <int D, typename T, int QB, int U>
__global__ void __launch_bounds__(NT)
    identify_multi_kernel(const CacheArgs c, const MethodArgs m, int layer_base,
                          uint8_t *label_out, int32_t *nh_out, float qscale, int max_len) {
  constexpr int RB = D * (int)sizeof(T);
  constexpr int EPL = Elem<T>::kPerPiece;
  constexpr int LPR = RB / 16;
  constexpr int RPW = 32 / LPR;
  constexpr int NW = NT / 32;
  extern __shared__ float e[];      // [QB][max_len] the pass's logits, then weights
  float *pbar = e + QB * max_len;  // [max_len] summed weights of all queries
  __shared__ float red[QB * NW];
  __shared__ float s_b[QB];
  __shared__ float fscan[33];
  __shared__ int s_nh;
  pdl_wait();
  pdl_launch_dependents();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int hl = blockIdx.x, i = layer_base + hl;
  const int len = c.len[i];
  const int ntok = c.ntok[i];
  const long long off = c.off[i];
  if (c.label[i] != HKV_DENSE || ntok <= 0) {  // in position order, with buffered queries
    if (tid == 0) set_err(c.err, HKV_ERR_STATE);
    return;
  }
  if (off < 0 || len <= 0 || off + len > c.arena_tokens) {
    if (tid == 0) set_err(c.err, HKV_ERR_BOUNDS);
    return;
  }
  if (len > max_len) {
    if (tid == 0) set_err(c.err, HKV_ERR_CAPACITY);
    return;
  }
  const int Pe = min(m.P, min(ntok, len));
  const int grp = lane / LPR, col = lane % LPR;
  const unsigned char *K = static_cast<const unsigned char *>(c.K) + off * RB;
  const unsigned char *ring = static_cast<const unsigned char *>(c.qbuf) + (size_t)i * m.P * RB;
  for (int r = tid; r < len; r += NT) pbar[r] = 0.f;
  for (int p0 = 0; p0 < Pe; p0 += QB) {
    // query p0 + b sees mq[b] keys (0 past the newest query)
    int mq[QB];
    float qf[QB][EPL];
#pragma unroll
    for (int b = 0; b < QB; ++b) {
      const int p = p0 + b;
      mq[b] = p < Pe ? len - (Pe - 1 - p) : 0;
#pragma unroll
      for (int x = 0; x < EPL; ++x) qf[b][x] = 0.f;
      if (p < Pe) {
        const int slot = (ntok - Pe + p) % m.P;
        Elem<T>::unpack(*reinterpret_cast<const uint4 *>(ring + (size_t)slot * RB + col * 16),
                        qf[b]);
#pragma unroll
        for (int x = 0; x < EPL; ++x) qf[b][x] *= qscale;
      }
    }
    const int mmax = len - max(0, Pe - 1 - (p0 + QB - 1));  // keys of the pass's newest query
    // logits (log2 units); U row steps load before any is used
    for (int r0 = warp * RPW; r0 < mmax; r0 += U * NW * RPW) {
      uint4 kr[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int r = r0 + u * NW * RPW + grp;
        kr[u] = r < mmax ? *reinterpret_cast<const uint4 *>(K + (size_t)r * RB + col * 16)
                         : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int r = r0 + u * NW * RPW + grp;
        float kf[EPL];
        Elem<T>::unpack(kr[u], kf);
        float dot[QB];
#pragma unroll
        for (int b = 0; b < QB; ++b) {
          dot[b] = 0.f;
#pragma unroll
          for (int x = 0; x < EPL; ++x) dot[b] = fmaf(qf[b][x], kf[x], dot[b]);
        }
#pragma unroll
        for (int b = 0; b < QB; ++b) {
#pragma unroll
          for (int o = LPR / 2; o >= 1; o >>= 1) dot[b] += __shfl_xor_sync(0xFFFFFFFFu, dot[b], o);
          if (col == 0 && r < mq[b]) e[b * max_len + r] = dot[b];
        }
      }
    }
    __syncthreads();
    float acc[QB];
#pragma unroll
    for (int b = 0; b < QB; ++b) acc[b] = -INFINITY;
    for (int r = tid; r < mmax; r += NT)
#pragma unroll
      for (int b = 0; b < QB; ++b)
        if (r < mq[b]) acc[b] = fmaxf(acc[b], e[b * max_len + r]);
    block_all<true, QB>(acc, red, s_b);
    float mx[QB];
#pragma unroll
    for (int b = 0; b < QB; ++b) {
      mx[b] = acc[b];
      acc[b] = 0.f;
    }
    for (int r = tid; r < mmax; r += NT)
#pragma unroll
      for (int b = 0; b < QB; ++b)
        if (r < mq[b]) {
          const float x = exp2f(e[b * max_len + r] - mx[b]);
          e[b * max_len + r] = x;
          acc[b] += x;
        }
    block_all<false, QB>(acc, red, s_b);
#pragma unroll
    for (int b = 0; b < QB; ++b) acc[b] = 1.f / acc[b];  // unused past the newest query
    for (int r = tid; r < mmax; r += NT) {
      float s = pbar[r];
#pragma unroll
      for (int b = 0; b < QB; ++b)
        if (r < mq[b]) s = fmaf(e[b * max_len + r], acc[b], s);
      pbar[r] = s;
    }
    __syncthreads();  // e is rewritten by the next pass
  }
  float tot[1] = {0.f};
  for (int r = tid; r < len; r += NT) tot[0] += pbar[r];
  block_all<false, 1>(tot, red, s_b);
  const float thr = tot[0] * m.tau;
  if (tid == 0) s_nh = len;
  __syncthreads();
  int *perm = nullptr;
  if (m.grid2d) {
    unsigned char *base =
        reinterpret_cast<unsigned char *>(e) + id_order_offset((size_t)(QB + 1) * max_len);
    perm = reinterpret_cast<int *>(base + (size_t)max_len * 8);
    grid_count_order(c.pos + off, len, m.C, m.row_len, ntok - 1,
                     reinterpret_cast<unsigned long long *>(base), perm);
  }
  float running = 0.f;  // cumulative mass from the newest token
  for (int base = 0; base < len; base += NT) {
    const int jb = base + tid;  // jb-th token counted (0 = current)
    const float x = jb < len ? pbar[perm ? perm[jb] : len - 1 - jb] : 0.f;
    float t;
    const float cum = running + block_excl_scan<float>(x, fscan, &t) + x;
    if (jb < len && cum >= thr) atomicMin(&s_nh, jb + 1);
    running += t;
  }
  __syncthreads();
  if (tid == 0) {
    label_out[i] = s_nh < m.w_loc ? HKV_LOCAL : HKV_GLOBAL;
    if (nh_out) nh_out[i] = s_nh;
  }
}

// Sec. 5.1 budgets (group = 0), or the aggregate-preserving variant over
// consecutive groups of `group` heads, one (sequence, layer) each: the
// (group - n_g)(B_g - w) tokens the local heads leave go to the group's n_g
// global heads in equal shares, the remainder one each to the global heads
// of lowest index.
__global__ void budgets_kernel(const uint8_t *label, int32_t *budget, int32_t *cap, int64_t *off,
                               int n, int C, int B_g, int w, int P, int group) {
  __shared__ long long scratch[33];
  pdl_wait();
  pdl_launch_dependents();
  long long running = 0;
  int bad = 0;
  for (int base = 0; base < n; base += blockDim.x) {
    const int i = base + threadIdx.x;
    long long cp = 0;
    if (i < n) {
      const uint8_t lb = label[i];
      int bg = 0;
      if (lb == HKV_GLOBAL) bg = B_g;
      else if (lb == HKV_LOCAL) bg = w;
      else bad = 1;
      if (group > 0 && lb == HKV_GLOBAL) {
        const int g0 = i / group * group;
        int ng = 0, rank = 0;
        for (int j = g0; j < g0 + group && j < n; ++j) {
          const bool gl = label[j] == HKV_GLOBAL;
          ng += gl;
          rank += gl && j < i;
        }
        const long long extra = (long long)(group - ng) * (B_g - w);
        bg += (int)(extra / ng) + (rank < extra % ng ? 1 : 0);
      }
      cp = (long long)C + bg + P;
      budget[i] = bg;
      cap[i] = (int32_t)cp;
    }
    long long tot;
    const long long ex = block_excl_scan<long long>(cp, scratch, &tot);
    if (i < n) off[i] = running + ex;
    running += tot;
  }
  if (__syncthreads_or(bad) && threadIdx.x == 0) off[n - 1] = -1;  // reported as a state error
}

}  // namespace

#ifdef HKV_UPD_TRACE
// tracer builds only: where the update's phase timestamps go
extern "C" int hkv_debug_set_utrace(unsigned long long *buf) {
  return cudaMemcpyToSymbol(g_utrace, &buf, sizeof(buf)) == cudaSuccess ? 0 : 7;
}
#endif

namespace {

template <int D, typename T>
cudaError_t prepare_t(size_t smem) {
  cudaError_t e = cudaFuncSetAttribute(append_evict_kernel<D, T>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(evict_kernel<D, T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(repack_kernel<D, T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
  const void *ident[] = {(const void *)identify_kernel<D, T, 2>,
                         (const void *)identify_kernel<D, T, 8>,
                         (const void *)identify_multi_kernel<D, T, 4, 2>,
                         (const void *)identify_multi_kernel<D, T, 4, 4>,
                         (const void *)identify_multi_kernel<D, T, 8, 2>,
                         (const void *)identify_multi_kernel<D, T, 8, 4>};
  for (const void *f : ident)
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  // all of an SM's L1 as shared memory, so that every head of a layer (one
  // CTA each) is resident at once
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(evict_kernel<D, T>, cudaFuncAttributePreferredSharedMemoryCarveout,
                             100);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(append_evict_kernel<D, T>,
                             cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  return e;
}

#define HKV_DISPATCH(D_, DT_, ...)                  \
  do {                                              \
    if ((DT_) == HKV_BF16) {                        \
      if ((D_) == 64) {                             \
        constexpr int kD = 64;                      \
        using kT = __nv_bfloat16;                   \
        __VA_ARGS__;                                \
      } else {                                      \
        constexpr int kD = 128;                     \
        using kT = __nv_bfloat16;                   \
        __VA_ARGS__;                                \
      }                                             \
    } else {                                        \
      if ((D_) == 64) {                             \
        constexpr int kD = 64;                      \
        using kT = float;                           \
        __VA_ARGS__;                                \
      } else {                                      \
        constexpr int kD = 128;                     \
        using kT = float;                           \
        __VA_ARGS__;                                \
      }                                             \
    }                                               \
  } while (0)

// launch with programmatic stream serialisation (the kernels wait for their
// predecessor with griddepcontrol.wait before touching memory)
template <typename... KArgs, typename... Args>
cudaError_t pdl_launch(void (*kernel)(KArgs...), int grid, int block, size_t smem, cudaStream_t s,
                       Args... args) {
  static const bool pdl = getenv("HKV_NO_PDL") == nullptr;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

size_t smem_of(int max_len, int D, int P, int es) {
  // the query ring / score stage; keys (8 B), positions (4 B), class/flag/
  // rank (4 B) per row; q-bar; two 256-bin histograms
  return ring_bytes(P, D, es, max_len) + (size_t)max_len * 16 + (size_t)D * 4 + 512 * 4 + 64;
}

// the longest segment a launch with `smem` bytes takes (the inverse of
// smem_of, which grows with max_len)
int max_len_of(size_t smem, int D, int P, int es) {
  int lo = 0, hi = 1 << 20;
  while (lo < hi) {
    const int mid = lo + (hi - lo + 1) / 2;
    if (smem_of(mid, D, P, es) <= smem) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

}  // namespace

size_t update_smem_bytes(int max_len, int D, int P, int dtype) {
  return smem_of(max_len, D, P, dtype == HKV_BF16 ? 2 : 4);
}

cudaError_t update_prepare(int D, int dtype, size_t smem) {
  HKV_DISPATCH(D, dtype, return prepare_t<kD, kT>(smem));
  return cudaErrorInvalidValue;
}

cudaError_t launch_append_evict(const CacheArgs &c, const MethodArgs &m, int layer_base,
                                int nheads, const void *q, const void *k, const void *v, int D,
                                int dtype, size_t smem, cudaStream_t s) {
  const int max_len = max_len_of(smem, D, m.P, dtype == HKV_BF16 ? 2 : 4);
  HKV_DISPATCH(D, dtype,
               return pdl_launch(append_evict_kernel<kD, kT>, nheads, NT, smem, s, c, m,
                                 layer_base, q, k, v, max_len));
  return cudaErrorInvalidValue;
}

cudaError_t launch_evict(const CacheArgs &c, const MethodArgs &m, int layer_base, int nheads,
                         int D, int dtype, size_t smem, cudaStream_t s) {
  const int max_len = max_len_of(smem, D, m.P, dtype == HKV_BF16 ? 2 : 4);
  HKV_DISPATCH(D, dtype,
               return pdl_launch(evict_kernel<kD, kT>, nheads, NT, smem, s, c, m, layer_base,
                                 max_len));
  return cudaErrorInvalidValue;
}

cudaError_t launch_repack(const CacheArgs &dense, const CacheArgs &ragged, const MethodArgs &m,
                          int layer_base, int nheads, int D, int dtype, size_t smem,
                          cudaStream_t s) {
  const int max_len = max_len_of(smem, D, m.P, dtype == HKV_BF16 ? 2 : 4);
  HKV_DISPATCH(D, dtype,
               return pdl_launch(repack_kernel<kD, kT>, nheads, NT, smem, s, dense, ragged, m,
                                 layer_base, max_len));
  return cudaErrorInvalidValue;
}

cudaError_t launch_prefill(const CacheArgs &c, int layer_base, int nheads, int C, const void *kc,
                           const void *vc, int D, int dtype, cudaStream_t s) {
  HKV_DISPATCH(D, dtype,
               return pdl_launch(prefill_kernel<kD, kT>, nheads, 128, 0, s, c, layer_base, C, kc,
                                 vc));
  return cudaErrorInvalidValue;
}

cudaError_t launch_init_dense(const CacheArgs &c, int n, int seg, cudaStream_t s) {
  int grid = (n + 255) / 256;
  if (grid > 4096) grid = 4096;
  if (grid < 1) grid = 1;
  return pdl_launch(init_dense_kernel, grid, 256, 0, s, c, n, seg);
}

cudaError_t launch_identify(const CacheArgs &c, const MethodArgs &m, int layer_base, int nheads,
                            const void *q, uint8_t *label_out, int32_t *nh_out, int D, int dtype,
                            int max_len, cudaStream_t s) {
  const float qscale = (float)(1.4426950408889634 / sqrt((double)D));
  const size_t smem = identify_smem_bytes(max_len, m.P, m.grid2d != 0, false);
  if (id_rows_in_flight(max_len, false) == 8) {
    HKV_DISPATCH(D, dtype,
                 return pdl_launch(identify_kernel<kD, kT, 8>, nheads, NT, smem, s, c, m,
                                   layer_base, q, label_out, nh_out, qscale, max_len));
  }
  HKV_DISPATCH(D, dtype,
               return pdl_launch(identify_kernel<kD, kT, 2>, nheads, NT, smem, s, c, m, layer_base,
                                 q, label_out, nh_out, qscale, max_len));
  return cudaErrorInvalidValue;
}

cudaError_t launch_identify_multi(const CacheArgs &c, const MethodArgs &m, int layer_base,
                                  int nheads, uint8_t *label_out, int32_t *nh_out, int D,
                                  int dtype, int max_len, cudaStream_t s) {
  const float qscale = (float)(1.4426950408889634 / sqrt((double)D));
  const size_t smem = identify_smem_bytes(max_len, m.P, m.grid2d != 0, true);
  const bool q8 = id_qb(m.P) == 8, u4 = id_rows_in_flight(max_len, true) == 4;
#define HKV_ID_MULTI(QB_, U_)                                                                  \
  HKV_DISPATCH(D, dtype,                                                                       \
               return pdl_launch(identify_multi_kernel<kD, kT, QB_, U_>, nheads, NT, smem, s, c, \
                                 m, layer_base, label_out, nh_out, qscale, max_len))
  if (q8 && u4) HKV_ID_MULTI(8, 4);
  if (q8) HKV_ID_MULTI(8, 2);
  if (u4) HKV_ID_MULTI(4, 4);
  HKV_ID_MULTI(4, 2);
#undef HKV_ID_MULTI
  return cudaErrorInvalidValue;
}

size_t identify_smem_bytes(int max_len, int P, bool grid2d, bool multi) {
  const size_t floats = multi ? (size_t)(id_qb(P) + 1) * max_len : (size_t)max_len;
  return id_smem(floats, max_len, grid2d);
}

cudaError_t launch_budgets(const uint8_t *label, int32_t *budget, int32_t *cap, int64_t *off,
                           int n, int C, int B_g, int w, int P, int group, cudaStream_t s) {
  return pdl_launch(budgets_kernel, 1, 1024, 0, s, label, budget, cap, off, n, C, B_g, w, P, group);
}

}  // namespace hkv
