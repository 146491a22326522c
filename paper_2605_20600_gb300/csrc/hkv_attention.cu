// Single-query decode attention over a ragged per-head KV cache (HeadKV,
// Eq. 1 applied to each head's retained tokens).
//
// Design (GB300, memory bound: every retained K/V byte is read once):
//  * split-K over the layer's TOTAL token count: the concatenation of all
//    heads' live tokens is cut into gridDim.x equal contiguous ranges, so
//    local heads (short) and global heads (long) load-balance exactly; a
//    range may cover the end of one head, whole heads, and the start of
//    another;
//  * K/V tiles of 8 KB each are staged into shared memory by the TMA engine
//    (1D cp.async.bulk, completion on an mbarrier), 4 stages deep;
//  * each warp takes whole token rows with 16-byte lanes (a 256-byte bf16
//    row is 16 lanes), a shuffle-xor tree per row for q.k, online softmax in
//    the log2 domain with fp32 accumulation;
//  * a head split across CTAs is combined by the last CTA to arrive (per-head
//    atomic counter, no spinning); partials are merged in CTA order, so the
//    result does not depend on arrival order.
#include <math.h>

#include "hkv_device.cuh"
#include "hkv_kernels.h"

namespace hkv {
namespace {

template <int D, typename T>
struct AttnShape {
  static constexpr int kES = sizeof(T);
  static constexpr int kRB = D * kES;             // bytes per token row
  static constexpr int kLPR = kRB / 16;           // lanes per row
  static constexpr int kEPL = 16 / kES;           // elements per lane
  static constexpr int kRPW = 32 / kLPR;          // rows per warp step
  static constexpr int kNW = kAttnThreads / 32;   // warps
  static constexpr int kTT = 8192 / kRB;          // rows per tile
  static constexpr int kSteps = kTT / (kNW * kRPW);
  static constexpr int kNS = 4;                   // pipeline stages
  static constexpr int kStageBytes = 2 * kTT * kRB;
  static constexpr int kMinChunk = 2 * kTT;       // fewest tokens per CTA
  static_assert(kLPR >= 1 && kLPR <= 32 && 32 % kLPR == 0, "row mapping");
  static_assert(kSteps >= 1 && kTT % (kNW * kRPW) == 0, "tile mapping");
  static_assert(D <= kAttnThreads, "one thread per output channel");
};

// Walks the tiles of one CTA's token range [g, b) head by head.
struct TileIter {
  int h;         // current head (layer-local index)
  int hl;        // its live length
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
  __device__ __forceinline__ void advance(int tt, const int32_t *len, int nheads) {
    g = tile_end(tt);
    if (g >= b) return;
    while (g >= hs + hl) {  // next head holding token g (skips empty heads)
      hs += hl;
      ++h;
      hl = h < nheads ? len[h] : 0;
    }
  }
};

template <int D, typename T>
__global__ void __launch_bounds__(kAttnThreads) attn_kernel(const AttnArgs p) {
  using S = AttnShape<D, T>;
  constexpr int NW = S::kNW, LPR = S::kLPR, EPL = S::kEPL, RPW = S::kRPW, TT = S::kTT;
  constexpr int RB = S::kRB, NS = S::kNS;

  extern __shared__ __align__(128) unsigned char stages[];
  __shared__ uint64_t bars[NS];
  __shared__ float red_acc[NW][D];
  __shared__ float red_m[NW], red_l[NW];
  __shared__ long long scan_scratch[33];
  __shared__ int s_h0, s_last;
  __shared__ long long s_hs0;

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nheads = p.nheads;

  // ---- pass 1: total live tokens of the layer, segment bounds -------------
  long long total = 0;
  int bad = 0;
  for (int base = 0; base < nheads; base += kAttnThreads) {
    const int h = base + tid;
    long long L = 0;
    if (h < nheads) {
      const int l = p.len[h];
      const long long o = p.off[h];
      if (l < 0 || o < 0 || o + l > p.arena_tokens) bad = 1;
      else L = l;
      if (l == 0 && blockIdx.x == 0)  // empty head: defined as zeros
        for (int d = 0; d < D; ++d) p.out[(size_t)h * D + d] = 0.f;
    }
    long long tot;
    block_excl_scan<long long>(L, scan_scratch, &tot);
    total += tot;
  }
  if (__syncthreads_or(bad)) {
    if (blockIdx.x == 0 && tid == 0) set_err(p.err, HKV_ERR_BOUNDS);
    return;
  }
  long long chunk = (total + gridDim.x - 1) / gridDim.x;
  if (chunk < S::kMinChunk) chunk = S::kMinChunk;
  const long long a = (long long)blockIdx.x * chunk;
  if (a >= total) return;
  const long long b = a + chunk < total ? a + chunk : total;

  // ---- pass 2: the head holding token a -----------------------------------
  {
    long long run = 0;
    for (int base = 0; base < nheads; base += kAttnThreads) {
      const int h = base + tid;
      const long long L = h < nheads ? p.len[h] : 0;
      long long tot;
      const long long st = run + block_excl_scan<long long>(L, scan_scratch, &tot);
      if (L > 0 && st <= a && a < st + L) {
        s_h0 = h;
        s_hs0 = st;
      }
      run += tot;
      if (run > a) break;  // uniform: every thread holds the same run
    }
  }
  if (tid == 0) {
    for (int s = 0; s < NS; ++s) mbar_init(&bars[s], 1);
    fence_barrier_init();
  }
  __syncthreads();

  TileIter cit;
  cit.h = s_h0;
  cit.hs = s_hs0;
  cit.hl = p.len[cit.h];
  cit.g = a;
  cit.b = b;

  // ---- producer (thread 0): keeps NS tiles in flight ----------------------
  TileIter pit = cit;
  int issued = 0;
  auto issue = [&]() {
    const int stage = issued % NS;
    const long long ge = pit.tile_end(TT);
    const uint32_t bytes = (uint32_t)(ge - pit.g) * RB;
    const long long row = p.off[pit.h] + (pit.g - pit.hs);
    unsigned char *dk = stages + stage * S::kStageBytes;
    mbar_arrive_expect_tx(&bars[stage], 2 * bytes);
    bulk_g2s(dk, static_cast<const unsigned char *>(p.K) + row * RB, bytes, &bars[stage]);
    bulk_g2s(dk + TT * RB, static_cast<const unsigned char *>(p.V) + row * RB, bytes,
             &bars[stage]);
    pit.advance(TT, p.len, nheads);
    ++issued;
  };
  if (tid == 0)
    for (int s = 0; s < NS && !pit.done(); ++s) issue();

  // ---- consumers ----------------------------------------------------------
  const int grp = lane / LPR, col = lane % LPR;
  float q[EPL], acc[EPL];
  float m = -INFINITY, l = 0.f;
#pragma unroll
  for (int e = 0; e < EPL; ++e) acc[e] = 0.f;

  for (int tile = 0; !cit.done(); ++tile) {
    const int stage = tile % NS;
    const bool ok = mbar_wait(&bars[stage], (uint32_t)(tile / NS) & 1u);
    if (__syncthreads_or(!ok)) {
      if (tid == 0) {
        set_err(p.err, HKV_ERR_TIMEOUT);
        for (int j = tile; j < issued; ++j) mbar_wait(&bars[j % NS], (uint32_t)(j / NS) & 1u);
      }
      return;
    }
    // every thread is done with tile-1: its stage takes the next tile
    if (tid == 0 && tile >= 1 && !pit.done()) issue();

    const long long ge = cit.tile_end(TT);
    const int n = (int)(ge - cit.g);
    const long long he = cit.hs + cit.hl;
    if (cit.g == cit.hs || cit.g == a) {  // first tile of this head here
      const uint4 u = *reinterpret_cast<const uint4 *>(
          static_cast<const unsigned char *>(p.q) + (size_t)cit.h * RB + col * 16);
      Elem<T>::unpack(u, q);
#pragma unroll
      for (int e = 0; e < EPL; ++e) {
        q[e] *= p.qscale;
        acc[e] = 0.f;
      }
      m = -INFINITY;
      l = 0.f;
    }

    const unsigned char *Ks = stages + stage * S::kStageBytes;
    const unsigned char *Vs = Ks + TT * RB;
    float sc[S::kSteps];
#pragma unroll
    for (int st = 0; st < S::kSteps; ++st) {
      const int r = st * (NW * RPW) + warp * RPW + grp;
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
        const int r = st * (NW * RPW) + warp * RPW + grp;
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

    if (ge == (b < he ? b : he)) {  // last tile of this head here: finish it
      // merge the row groups of the warp
#pragma unroll
      for (int o = LPR; o < 32; o <<= 1) {
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
      if (lane < LPR) {
#pragma unroll
        for (int e = 0; e < EPL; ++e) red_acc[warp][lane * EPL + e] = acc[e];
        if (lane == 0) {
          red_m[warp] = m;
          red_l[warp] = l;
        }
      }
      __syncthreads();
      const int h = cit.h;
      const long long hs = cit.hs;
      const bool whole = hs >= a && he <= b;
      if (tid < D) {
        float mx = red_m[0];
#pragma unroll
        for (int w = 1; w < NW; ++w) mx = fmaxf(mx, red_m[w]);
        float L = 0.f, A = 0.f;
#pragma unroll
        for (int w = 0; w < NW; ++w) {
          const float s = red_m[w] == -INFINITY ? 0.f : exp2f(red_m[w] - mx);
          L += red_l[w] * s;
          A += red_acc[w][tid] * s;
        }
        if (whole) {
          p.out[(size_t)h * D + tid] = A / L;
        } else {
          float *pp = p.part + ((size_t)blockIdx.x * 2 + (hs <= a ? 0 : 1)) * (D + 2);
          pp[tid] = A;
          if (tid == 0) {
            pp[D] = mx;
            pp[D + 1] = L;
          }
        }
      }
      if (!whole) {
        __threadfence();
        __syncthreads();
        const long long c0 = hs / chunk, c1 = (he - 1) / chunk;
        if (tid == 0) s_last = atomicAdd(&p.cnt[h], 1) == (int)(c1 - c0);
        __syncthreads();
        if (s_last) {
          __threadfence();
          if (tid < D) {
            float mx = -INFINITY;
            for (long long c = c0; c <= c1; ++c) {
              const int slot = (c == c0 && c * chunk < hs) ? 1 : 0;
              mx = fmaxf(mx, __ldcg(p.part + ((size_t)c * 2 + slot) * (D + 2) + D));
            }
            float L = 0.f, A = 0.f;
            for (long long c = c0; c <= c1; ++c) {
              const int slot = (c == c0 && c * chunk < hs) ? 1 : 0;
              const float *pp = p.part + ((size_t)c * 2 + slot) * (D + 2);
              const float s = exp2f(__ldcg(pp + D) - mx);
              L += __ldcg(pp + D + 1) * s;
              A += __ldcg(pp + tid) * s;
            }
            p.out[(size_t)h * D + tid] = A / L;
          }
          if (tid == 0) p.cnt[h] = 0;
        }
      }
      __syncthreads();
    }
    cit.advance(TT, p.len, nheads);
  }
}

template <int D, typename T>
size_t smem_bytes() {
  return (size_t)AttnShape<D, T>::kNS * AttnShape<D, T>::kStageBytes;
}

template <int D, typename T>
cudaError_t prepare_t(int *ctas) {
  const size_t smem = smem_bytes<D, T>();
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<D, T>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(ctas, attn_kernel<D, T>, kAttnThreads,
                                                       smem);
}

template <int D, typename T>
cudaError_t launch_t(const AttnArgs &a, int grid, cudaStream_t s) {
  attn_kernel<D, T><<<grid, kAttnThreads, smem_bytes<D, T>(), s>>>(a);
  return cudaGetLastError();
}

}  // namespace

size_t attention_smem_bytes(int D, int dtype) {
  if (dtype == HKV_BF16) return D == 64 ? smem_bytes<64, __nv_bfloat16>() : smem_bytes<128, __nv_bfloat16>();
  return D == 64 ? smem_bytes<64, float>() : smem_bytes<128, float>();
}

cudaError_t attention_prepare(int D, int dtype, int *ctas) {
  if (dtype == HKV_BF16) return D == 64 ? prepare_t<64, __nv_bfloat16>(ctas) : prepare_t<128, __nv_bfloat16>(ctas);
  return D == 64 ? prepare_t<64, float>(ctas) : prepare_t<128, float>(ctas);
}

cudaError_t launch_attention(const AttnArgs &a, int D, int dtype, int grid, cudaStream_t s) {
  if (dtype == HKV_BF16)
    return D == 64 ? launch_t<64, __nv_bfloat16>(a, grid, s) : launch_t<128, __nv_bfloat16>(a, grid, s);
  return D == 64 ? launch_t<64, float>(a, grid, s) : launch_t<128, float>(a, grid, s);
}

}  // namespace hkv
