// Device code shared by the two decode-step designs (hkv_attention.cu: an
// attention kernel plus a finishing kernel; hkv_step.cu: one kernel that
// also merges split heads and advances the counters): tile shapes, the
// consumers' per-lane arithmetic, the tile iterator and the programmatic
// dependent launch controls.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "hkv_device.cuh"

namespace hkv {
namespace {

// Tuning knobs (compile time), per head dimension: consumer warps, bytes of
// K per pipeline stage and stages (measured: rows of 256 B stream best with 7
// consumer warps over 10.5 KB tiles in 4 stages; rows of 128 B, whose short
// heads come many to a CTA, with 8 warps over 8 KB tiles in 5 stages); a cap
// on resident CTAs per SM used to size the grid, and tiles loaded before the
// wait for the previous kernel (prefetch).
#ifndef HKV_ATTN_CW_D128
#define HKV_ATTN_CW_D128 7
#endif
#ifndef HKV_ATTN_TILE_BYTES_D128
#define HKV_ATTN_TILE_BYTES_D128 10752
#endif
#ifndef HKV_ATTN_STAGES_D128
#define HKV_ATTN_STAGES_D128 4
#endif
#ifndef HKV_ATTN_CW_D64
#define HKV_ATTN_CW_D64 8
#endif
#ifndef HKV_ATTN_TILE_BYTES_D64
#define HKV_ATTN_TILE_BYTES_D64 8192
#endif
#ifndef HKV_ATTN_STAGES_D64
#define HKV_ATTN_STAGES_D64 5
#endif
#ifndef HKV_ATTN_MAX_CTAS_PER_SM
#define HKV_ATTN_MAX_CTAS_PER_SM 2
#endif
#ifndef HKV_ATTN_PRE_TILES
#define HKV_ATTN_PRE_TILES 3
#endif

// Tile and pipeline shape of a decode kernel: CW consumer warps, TB bytes of
// K per stage, NSTG stages, PRE tiles loaded before the dependency wait.
template <int D, typename T, int CW, int TB, int NSTG, int PRE>
struct TileShape {
  static constexpr int kCW = CW;                  // consumer warps
  static constexpr int kThreads = 32 * (kCW + 2);  // + producer + epilogue
  static constexpr int kES = sizeof(T);
  static constexpr int kRB = D * kES;             // bytes per token row
  static constexpr int kLPR = kRB / 16;           // lanes per row
  static constexpr int kEPL = 16 / kES;           // elements per lane
  static constexpr int kRPW = 32 / kLPR;          // rows per warp step
  static constexpr int kTT =                      // rows per tile
      TB / kRB;
  static constexpr int kSteps = kTT / (kCW * kRPW);
  static constexpr int kNS = NSTG;                // stages
  static constexpr int kPre = PRE;                // tiles loaded before the wait
  static constexpr int kStageBytes = 2 * kTT * kRB + kRB;   // K, V, q row
  static constexpr int kMinChunk = 2 * kTT;       // fewest indices per CTA range
  static_assert(kLPR >= 1 && kLPR <= 32 && 32 % kLPR == 0, "row mapping");
  static_assert(kSteps >= 1 && kTT % (kCW * kRPW) == 0, "tile mapping");
  static_assert(D <= kCW * 32 && D % 32 == 0, "output channels");
  static_assert(kStageBytes % 16 == 0, "TMA alignment");
  static_assert(PRE >= 0 && PRE <= kNS, "prefetch depth");
};

// the two-kernel design's shape (hkv_attention.cu)
template <int D, typename T>
using AttnShape =
    TileShape<D, T, D == 64 ? HKV_ATTN_CW_D64 : HKV_ATTN_CW_D128,
              D == 64 ? HKV_ATTN_TILE_BYTES_D64 : HKV_ATTN_TILE_BYTES_D128,
              D == 64 ? HKV_ATTN_STAGES_D64 : HKV_ATTN_STAGES_D128, HKV_ATTN_PRE_TILES>;

// N consecutive floats as one vector access (N = 2 or 4)
template <int N>
struct Vec;
template <>
struct Vec<4> {
  __device__ static __forceinline__ void st(float *p, const float *v) {
    *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
  }
  __device__ static __forceinline__ void lds(const float *p, float *v) {
    const float4 x = *reinterpret_cast<const float4 *>(p);
    v[0] = x.x, v[1] = x.y, v[2] = x.z, v[3] = x.w;
  }
  __device__ static __forceinline__ void ldcg(const float *p, float *v) {
    const float4 x = __ldcg(reinterpret_cast<const float4 *>(p));
    v[0] = x.x, v[1] = x.y, v[2] = x.z, v[3] = x.w;
  }
};
template <>
struct Vec<2> {
  __device__ static __forceinline__ void st(float *p, const float *v) {
    *reinterpret_cast<float2 *>(p) = make_float2(v[0], v[1]);
  }
  __device__ static __forceinline__ void lds(const float *p, float *v) {
    const float2 x = *reinterpret_cast<const float2 *>(p);
    v[0] = x.x, v[1] = x.y;
  }
  __device__ static __forceinline__ void ldcg(const float *p, float *v) {
    const float2 x = __ldcg(reinterpret_cast<const float2 *>(p));
    v[0] = x.x, v[1] = x.y;
  }
};

__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Head h of n rows takes slot_len(n) indices: whole tiles of TT rows, the
// last one partly filled.
template <int TT>
__device__ __forceinline__ long long slot_len(long long n) {
  return (n + TT - 1) / TT * TT;
}

// Walks the tiles of a slot-aligned range [g, b) of the index space head by
// head.
template <int TT>
struct TileIter {
  int h;         // current head (layer-local index)
  int hl;        // its (virtual) length
  long long hs;  // index where head h starts
  long long g;   // start of the current tile (a slot boundary)
  long long b;   // end of the range (a slot boundary)

  __device__ __forceinline__ bool done() const { return g >= b; }
  __device__ __forceinline__ long long tile_end() const {  // end of the tile's rows
    long long e = g + TT;
    const long long he = hs + hl;
    if (e > he) e = he;
    if (e > b) e = b;
    return e;
  }
  template <class L>
  __device__ __forceinline__ void advance(const L &look) {
    g += TT;
    if (g >= b) return;
    while (g >= hs + slot_len<TT>(hl)) {  // next head holding slot g (skips empty heads)
      hs += slot_len<TT>(hl);
      ++h;
      hl = look.vlen(h);
    }
  }
};

// The consumers' arithmetic on one 16-byte piece of a row.
//  * bf16: the query stays in its packed pairs and q.k takes one
//    mixed-precision FMA per element (a bf16 x bf16 product is exact in
//    fp32, so this equals widening first); the scale goes on the sum;
//  * fp32: the query is scaled when loaded;
//  * V rows accumulate into fp32 pairs with paired FMAs.
template <typename T>
struct LaneMath;
template <>
struct LaneMath<__nv_bfloat16> {
  static constexpr int kEPL = 8;
  struct Q {
    uint32_t w[4];
  };
  __device__ static __forceinline__ void load_q(Q &q, const uint4 &u, float) {
    q.w[0] = u.x, q.w[1] = u.y, q.w[2] = u.z, q.w[3] = u.w;
  }
  __device__ static __forceinline__ void fma_pair(float &d0, float &d1, uint32_t a, uint32_t b) {
    asm("{\n\t.reg .b16 al, ah, bl, bh;\n\t"
        "mov.b32 {al, ah}, %2;\n\t"
        "mov.b32 {bl, bh}, %3;\n\t"
        "fma.rn.f32.bf16 %0, al, bl, %0;\n\t"
        "fma.rn.f32.bf16 %1, ah, bh, %1;\n\t}"
        : "+f"(d0), "+f"(d1)
        : "r"(a), "r"(b));
  }
  __device__ static __forceinline__ float dot(const Q &q, const uint4 &k) {
    float d0 = 0.f, d1 = 0.f;
    fma_pair(d0, d1, q.w[0], k.x);
    fma_pair(d0, d1, q.w[1], k.y);
    fma_pair(d0, d1, q.w[2], k.z);
    fma_pair(d0, d1, q.w[3], k.w);
    return d0 + d1;
  }
  __device__ static __forceinline__ float score(float dot, float qscale) { return dot * qscale; }
  __device__ static __forceinline__ float2 widen(uint32_t w) {
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
  }
  __device__ static __forceinline__ void add_v(float2 *acc, const uint4 &v, float pr) {
    const float2 p2 = make_float2(pr, pr);
    acc[0] = __ffma2_rn(widen(v.x), p2, acc[0]);
    acc[1] = __ffma2_rn(widen(v.y), p2, acc[1]);
    acc[2] = __ffma2_rn(widen(v.z), p2, acc[2]);
    acc[3] = __ffma2_rn(widen(v.w), p2, acc[3]);
  }
};
template <>
struct LaneMath<float> {
  static constexpr int kEPL = 4;
  struct Q {
    float f[4];
  };
  __device__ static __forceinline__ void load_q(Q &q, const uint4 &u, float qscale) {
    q.f[0] = __uint_as_float(u.x) * qscale;
    q.f[1] = __uint_as_float(u.y) * qscale;
    q.f[2] = __uint_as_float(u.z) * qscale;
    q.f[3] = __uint_as_float(u.w) * qscale;
  }
  __device__ static __forceinline__ float dot(const Q &q, const uint4 &k) {
    const float d0 = fmaf(q.f[2], __uint_as_float(k.z), q.f[0] * __uint_as_float(k.x));
    const float d1 = fmaf(q.f[3], __uint_as_float(k.w), q.f[1] * __uint_as_float(k.y));
    return d0 + d1;
  }
  __device__ static __forceinline__ float score(float dot, float) { return dot; }
  __device__ static __forceinline__ void add_v(float2 *acc, const uint4 &v, float pr) {
    const float2 p2 = make_float2(pr, pr);
    acc[0] = __ffma2_rn(make_float2(__uint_as_float(v.x), __uint_as_float(v.y)), p2, acc[0]);
    acc[1] = __ffma2_rn(make_float2(__uint_as_float(v.z), __uint_as_float(v.w)), p2, acc[1]);
  }
};

}  // namespace
}  // namespace hkv
