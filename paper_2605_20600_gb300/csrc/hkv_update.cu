// Per-head cache maintenance of HeadKV, one CTA per head:
//  * append_evict: the periodic head-aware update when the buffer is full
//    (Sec. 4: local heads drop their history, Eq. 3; global heads trim it
//    by Stratified Token Eviction, Eqs. 4-6), then the append of the new
//    token (Sec. 3, KV Cache);
//  * repack: the first update at grouping, out of place from the dense
//    cache into the ragged one (Step 3);
//  * prefill / init_dense: the uncompressed cache of Step 1;
//  * identify: threshold-based attention accumulation (Step 2);
//  * budgets: per-head budgets and the arena layout (Sec. 5.1).
//
// STE on the device: the P buffered queries are summed (q-bar), each
// history key is scored q-bar . k in a fixed fp32 order, a (score, position)
// 64-bit key is formed (unique, ascending = evict first), an 8-pass radix
// select finds the quota-th smallest key of the long- and near-range
// subsets at once, and a block prefix sum over the keep flags gives every
// survivor its new row; rows move in ascending chunks (destination <=
// source), each chunk fully loaded before any of it is stored, so the
// compaction is safe in place.
#include <math.h>

#include "hkv_device.cuh"
#include "hkv_kernels.h"

namespace hkv {
namespace {

constexpr int NT = kCacheThreads;

struct SegRef {
  const unsigned char *sk, *sv;  // source rows, row 0 = segment start
  const int32_t *spos;
  unsigned char *dk, *dv;        // destination rows
  int32_t *dpos;
  int len;                       // live source rows
  int dst_cap;                   // destination capacity (rows)
  bool in_place;
};

struct SelectShared {
  unsigned long long prefix[2];
  int rem[2];
  int scan[33];
  int first;
  int bad;
};

// The k0-th smallest key among keys[0, n_long) and the k1-th among
// keys[n_long, T) (1-based; 0 = not needed), by MSD radix select on bytes.
// Keys are unique, so the result identifies exactly k keys at or below it.
__device__ void radix_select2(const unsigned long long *keys, int T, int n_long, int k0, int k1,
                              int *hist, SelectShared &sh) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (tid == 0) {
    sh.prefix[0] = sh.prefix[1] = 0ull;
    sh.rem[0] = k0;
    sh.rem[1] = k1;
  }
  __syncthreads();
  for (int shift = 56; shift >= 0; shift -= 8) {
    for (int i = tid; i < 512; i += NT) hist[i] = 0;
    __syncthreads();
    const unsigned long long hi = shift == 56 ? 0ull : (~0ull << (shift + 8));
    const unsigned long long p0 = sh.prefix[0], p1 = sh.prefix[1];
    const int r0 = sh.rem[0], r1 = sh.rem[1];
    for (int j = tid; j < T; j += NT) {
      const int s = j < n_long ? 0 : 1;
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
          int run = excl, digit = -1, rem = 0;
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            if (digit < 0 && run + c[e] >= target) {
              digit = lane * 8 + e;
              rem = target - run;
            }
            run += c[e];
          }
          sh.prefix[s] |= (unsigned long long)digit << shift;
          sh.rem[s] = rem;
        }
      }
    }
    __syncthreads();
  }
}

// One head-aware update of a segment (Eqs. 2-6). Returns the new length,
// or -1 if the destination is too small (error word set). Block-uniform.
template <int D, typename T>
__device__ int update_segment(const SegRef &sg, int label, const MethodArgs &m,
                              const unsigned char *qring, int ntok, unsigned char *dyn,
                              int max_len, uint32_t *err) {
  constexpr int RB = D * (int)sizeof(T);
  constexpr int EPL = Elem<T>::kPerPiece;
  constexpr int LPR = RB / 16;
  constexpr int U = 4;                 // 16-byte pieces per thread per chunk
  constexpr int CH = NT * U / LPR;     // rows per move chunk
  static_assert(CH <= NT, "one pos per thread per chunk");
  __shared__ SelectShared sh;

  const int tid = threadIdx.x;
  const int C = m.C;
  const int n_img = sg.len - C;
  const int n_recent = n_img < m.w ? n_img : m.w;
  const int NH = n_img - n_recent;  // history candidates (Eq. 2)
  int M = 0;
  if (label == HKV_LOCAL) M = NH;   // Eq. 3: no history
  else if (NH > m.hist_budget) M = NH - m.hist_budget;
  if (M == 0 && sg.in_place) return sg.len;
  if (sg.len - M > sg.dst_cap) {
    if (tid == 0) set_err(err, HKV_ERR_CAPACITY);
    return -1;
  }

  unsigned long long *keys = reinterpret_cast<unsigned long long *>(dyn);
  int *dst = reinterpret_cast<int *>(keys + max_len);
  float *qbar = reinterpret_cast<float *>(dst + max_len);
  int *hist = reinterpret_cast<int *>(qbar + D);

  // dst[] first holds the keep flags
  for (int r = tid; r < sg.len; r += NT) dst[r] = (r >= C && r < C + NH && label == HKV_LOCAL) ? 0 : 1;

  if (label == HKV_GLOBAL && M > 0) {
    // q-bar: the P buffered queries, oldest first (Eq. 6, reading R8/R10)
    const int P = m.P;
    for (int d = tid; d < D; d += NT) {
      float acc = 0.f;
      for (int pp = 0; pp < P; ++pp) {
        int slot = (ntok - P + pp) % P;
        if (slot < 0) slot += P;
        acc = __fadd_rn(acc, Elem<T>::load1(qring, (size_t)slot * D + d));
      }
      qbar[d] = acc;
    }
    __syncthreads();
    // scores s_j = q-bar . k_j, d ascending, each product and sum rounded
    for (int j = tid; j < NH; j += NT) {
      const unsigned char *krow = sg.sk + (size_t)(C + j) * RB;
      float s = 0.f;
#pragma unroll 4
      for (int pc = 0; pc < LPR; ++pc) {
        float kf[EPL];
        Elem<T>::unpack(*reinterpret_cast<const uint4 *>(krow + pc * 16), kf);
#pragma unroll
        for (int e = 0; e < EPL; ++e) s = __fadd_rn(s, __fmul_rn(qbar[pc * EPL + e], kf[e]));
      }
      s = __fadd_rn(s, 0.f);  // -0 reads as +0
      uint32_t u = __float_as_uint(s);
      u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);  // order-preserving
      keys[j] = ((unsigned long long)u << 32) | (uint32_t)sg.spos[C + j];
    }
    __syncthreads();
    // Eq. 5 split and the M/2 quotas, excess of a short subset to the other
    const int n_long = (int)floor((double)NH * m.r_s);
    int m_long = M / 2, m_near = M - M / 2;
    if (m_long > n_long) {
      m_near += m_long - n_long;
      m_long = n_long;
    }
    if (m_near > NH - n_long) {
      m_long += m_near - (NH - n_long);
      m_near = NH - n_long;
    }
    radix_select2(keys, NH, n_long, m_long, m_near, hist, sh);
    const unsigned long long thr0 = sh.prefix[0], thr1 = sh.prefix[1];
    for (int j = tid; j < NH; j += NT) {
      const bool ev = j < n_long ? (m_long > 0 && keys[j] <= thr0) : (m_near > 0 && keys[j] <= thr1);
      if (ev) dst[C + j] = 0;
    }
  }
  if (tid == 0) sh.first = sg.len;
  __syncthreads();

  // prefix sum of keep flags -> destination rows; first row that moves
  int running = 0;
  for (int base = 0; base < sg.len; base += NT) {
    const int r = base + tid;
    const int k = r < sg.len ? dst[r] : 0;
    int tot;
    const int ex = block_excl_scan<int>(k, sh.scan, &tot);
    if (r < sg.len) {
      const int d = k ? running + ex : -1;
      dst[r] = d;
      if (d != r) atomicMin(&sh.first, r);
    }
    running += tot;
  }
  __syncthreads();
  const int new_len = running;
  const int first = sg.in_place ? sh.first : 0;

  // move rows in ascending chunks: load the whole chunk, then store it
  for (int c0 = first; c0 < sg.len; c0 += CH) {
    uint4 kr[U], vr[U];
    int drow[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int piece = u * NT + tid;
      const int r = c0 + piece / LPR, col = piece % LPR;
      drow[u] = r < sg.len ? dst[r] : -1;
      if (drow[u] >= 0) {
        kr[u] = __ldcg(reinterpret_cast<const uint4 *>(sg.sk + (size_t)r * RB + col * 16));
        vr[u] = __ldcg(reinterpret_cast<const uint4 *>(sg.sv + (size_t)r * RB + col * 16));
      }
    }
    const int pr = c0 + tid;
    const int pd = (tid < CH && pr < sg.len) ? dst[pr] : -1;
    const int pv = pd >= 0 ? __ldcg(sg.spos + pr) : 0;
    __syncthreads();
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int piece = u * NT + tid;
      const int col = piece % LPR;
      if (drow[u] >= 0) {
        *reinterpret_cast<uint4 *>(sg.dk + (size_t)drow[u] * RB + col * 16) = kr[u];
        *reinterpret_cast<uint4 *>(sg.dv + (size_t)drow[u] * RB + col * 16) = vr[u];
      }
    }
    if (pd >= 0) sg.dpos[pd] = pv;
    __syncthreads();
  }
  return new_len;
}

template <int D, typename T>
__global__ void __launch_bounds__(NT)
    append_evict_kernel(const CacheArgs c, const MethodArgs m, int layer_base, const void *q,
                        const void *k, const void *v, int max_len) {
  constexpr int RB = D * (int)sizeof(T);
  extern __shared__ __align__(16) unsigned char dyn[];
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
    SegRef sg{K, V, pos, K, V, pos, len, cp, true};
    const int nl = update_segment<D, T>(sg, lab, m, qring, ntok, dyn, max_len, c.err);
    if (nl < 0) return;
    len = nl;
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
__global__ void __launch_bounds__(NT)
    repack_kernel(const CacheArgs dn, const CacheArgs rg, const MethodArgs m, int layer_base,
                  int max_len) {
  constexpr int RB = D * (int)sizeof(T);
  extern __shared__ __align__(16) unsigned char dyn[];
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
            false};
  const unsigned char *qring = static_cast<const unsigned char *>(dn.qbuf) + (size_t)i * m.P * RB;
  const int nl = update_segment<D, T>(sg, lab, m, qring, dn.ntok[i], dyn, max_len, rg.err);
  if (nl < 0) return;
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

// Step 2: attention of the current query over the key cache, accumulated
// backward from the newest token until tau; local iff fewer than w_loc
// tokens were needed.
template <int D, typename T>
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
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int hl = blockIdx.x, i = layer_base + hl;
  const int len = c.len[i];
  const long long off = c.off[i];
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
  // logits (log2 units)
  for (int r0 = warp * RPW; r0 < len; r0 += NW * RPW) {
    const int r = r0 + grp;
    float dot = 0.f;
    if (r < len) {
      float kf[EPL];
      Elem<T>::unpack(*reinterpret_cast<const uint4 *>(K + (size_t)r * RB + col * 16), kf);
#pragma unroll
      for (int x = 0; x < EPL; ++x) dot = fmaf(qf[x], kf[x], dot);
    }
#pragma unroll
    for (int o = LPR / 2; o >= 1; o >>= 1) dot += __shfl_xor_sync(0xFFFFFFFFu, dot, o);
    if (r < len && col == 0) e[r] = dot;
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
  // backward cumulative mass from the newest token
  float running = 0.f;
  for (int base = 0; base < len; base += NT) {
    const int jb = base + tid;  // jb-th newest token (0 = current)
    const float x = jb < len ? e[len - 1 - jb] : 0.f;
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

__global__ void budgets_kernel(const uint8_t *label, int32_t *budget, int32_t *cap, int64_t *off,
                               int n, int C, int B_g, int w, int P) {
  __shared__ long long scratch[33];
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

template <int D, typename T>
cudaError_t prepare_t(size_t smem) {
  cudaError_t e = cudaFuncSetAttribute(append_evict_kernel<D, T>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(repack_kernel<D, T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(identify_kernel<D, T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)smem);
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

}  // namespace

size_t update_smem_bytes(int max_len, int D) {
  // keys (8 B) + destinations (4 B) per row, q-bar, two 256-bin histograms
  return (size_t)max_len * 12 + (size_t)D * 4 + 512 * 4 + 64;
}

cudaError_t update_prepare(int D, int dtype, size_t smem) {
  HKV_DISPATCH(D, dtype, return prepare_t<kD, kT>(smem));
  return cudaErrorInvalidValue;
}

cudaError_t launch_append_evict(const CacheArgs &c, const MethodArgs &m, int layer_base,
                                int nheads, const void *q, const void *k, const void *v, int D,
                                int dtype, size_t smem, cudaStream_t s) {
  const int max_len = (int)((smem - (size_t)D * 4 - 512 * 4 - 64) / 12);
  HKV_DISPATCH(D, dtype,
               (append_evict_kernel<kD, kT><<<nheads, NT, smem, s>>>(c, m, layer_base, q, k, v,
                                                                    max_len)));
  return cudaGetLastError();
}

cudaError_t launch_repack(const CacheArgs &dense, const CacheArgs &ragged, const MethodArgs &m,
                          int layer_base, int nheads, int D, int dtype, size_t smem,
                          cudaStream_t s) {
  const int max_len = (int)((smem - (size_t)D * 4 - 512 * 4 - 64) / 12);
  HKV_DISPATCH(D, dtype,
               (repack_kernel<kD, kT><<<nheads, NT, smem, s>>>(dense, ragged, m, layer_base,
                                                              max_len)));
  return cudaGetLastError();
}

cudaError_t launch_prefill(const CacheArgs &c, int layer_base, int nheads, int C, const void *kc,
                           const void *vc, int D, int dtype, cudaStream_t s) {
  HKV_DISPATCH(D, dtype, (prefill_kernel<kD, kT><<<nheads, 128, 0, s>>>(c, layer_base, C, kc, vc)));
  return cudaGetLastError();
}

cudaError_t launch_init_dense(const CacheArgs &c, int n, int seg, cudaStream_t s) {
  int grid = (n + 255) / 256;
  if (grid > 4096) grid = 4096;
  if (grid < 1) grid = 1;
  init_dense_kernel<<<grid, 256, 0, s>>>(c, n, seg);
  return cudaGetLastError();
}

cudaError_t launch_identify(const CacheArgs &c, const MethodArgs &m, int layer_base, int nheads,
                            const void *q, uint8_t *label_out, int32_t *nh_out, int D, int dtype,
                            int max_len, cudaStream_t s) {
  const float qscale = (float)(1.4426950408889634 / sqrt((double)D));
  const size_t smem = (size_t)max_len * 4;
  HKV_DISPATCH(D, dtype,
               (identify_kernel<kD, kT><<<nheads, NT, smem, s>>>(c, m, layer_base, q, label_out,
                                                                nh_out, qscale, max_len)));
  return cudaGetLastError();
}

cudaError_t launch_budgets(const uint8_t *label, int32_t *budget, int32_t *cap, int64_t *off,
                           int n, int C, int B_g, int w, int P, cudaStream_t s) {
  budgets_kernel<<<1, 1024, 0, s>>>(label, budget, cap, off, n, C, B_g, w, P);
  return cudaGetLastError();
}

}  // namespace hkv
