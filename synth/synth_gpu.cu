// GPU twin of synth/gen.py: writes the same seeded synthetic q/k/v bits on
// the device so that full-size workloads need no host generation or upload.
// Every step mirrors the Python definition: SplitMix64 output number n,
// Irwin-Hall sum of its four 16-bit fields, one fp32 multiply by a scale,
// fp32 products/sums with explicit round-to-nearest intrinsics (no FMA
// contraction), then rounding to the storage dtype.
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace {

__device__ __forceinline__ uint64_t splitmix64(uint64_t seed, uint64_t n) {
  uint64_t z = seed + (n + 1ull) * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t counter(uint64_t tensor, uint64_t s, uint64_t l,
                                            uint64_t h, uint64_t tok, uint64_t d) {
  return (((((tensor * 1024ull + s) * 128ull + l) * 128ull + h) * 16384ull + tok) * 256ull) + d;
}

__device__ __forceinline__ float irwin_hall4(uint64_t u) {
  long long a = (long long)(u & 0xFFFFull) + (long long)((u >> 16) & 0xFFFFull) +
                (long long)((u >> 32) & 0xFFFFull) + (long long)((u >> 48) & 0xFFFFull);
  return __ll2float_rn(a - 131070ll);
}

__device__ __forceinline__ void store(void* base, size_t i, float x, int bf16) {
  if (bf16) reinterpret_cast<__nv_bfloat16*>(base)[i] = __float2bfloat16_rn(x);
  else reinterpret_cast<float*>(base)[i] = x;
}

// out[(((tt*nl + li)*S + s)*H + h)*D + d] for image tokens t0+tt, layers l0+li
__global__ void synth_image_kernel(void* q, void* k, void* v, int bf16,
                                   const float* __restrict__ pe, const float* __restrict__ cq,
                                   uint64_t seed, int S, int H, int D, int C, int row_len,
                                   int L, int l0, int nl, int t0, int nt, float ks, float vs) {
  const size_t total = (size_t)nt * nl * S * H * D;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    size_t r = i;
    const int d = (int)(r % D); r /= D;
    const int h = (int)(r % H); r /= H;
    const int s = (int)(r % S); r /= S;
    const int li = (int)(r % nl); r /= nl;
    const int tt = (int)r;
    const int l = l0 + li, t = t0 + tt;
    const uint64_t tok = (uint64_t)(C + t);
    const float p = pe[((size_t)(t / row_len) * row_len + (t % row_len)) * D + d];
    const float gq = irwin_hall4(splitmix64(seed, counter(0, s, l, h, tok, d)));
    const float gk = irwin_hall4(splitmix64(seed, counter(1, s, l, h, tok, d)));
    const float gv = irwin_hall4(splitmix64(seed, counter(2, s, l, h, tok, d)));
    const float c = cq[(size_t)l * H + h];
    store(q, i, __fadd_rn(__fmul_rn(c, p), __fmul_rn(gq, ks)), bf16);
    store(k, i, __fadd_rn(p, __fmul_rn(gk, ks)), bf16);
    store(v, i, __fmul_rn(gv, vs), bf16);
  }
  (void)L;
}

// kc/vc[((s*H + h)*C + j)*D + d] for the conditioning tokens of layer l
__global__ void synth_cond_kernel(void* kc, void* vc, int bf16, uint64_t seed, int S, int H,
                                  int D, int C, int l, float ks, float vs) {
  const size_t total = (size_t)S * H * C * D;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < total;
       i += (size_t)gridDim.x * blockDim.x) {
    size_t r = i;
    const int d = (int)(r % D); r /= D;
    const int j = (int)(r % C); r /= C;
    const int h = (int)(r % H); r /= H;
    const int s = (int)r;
    const float gk = irwin_hall4(splitmix64(seed, counter(1, s, l, h, (uint64_t)j, d)));
    const float gv = irwin_hall4(splitmix64(seed, counter(2, s, l, h, (uint64_t)j, d)));
    store(kc, i, __fmul_rn(gk, ks), bf16);
    store(vc, i, __fmul_rn(gv, vs), bf16);
  }
}

int grid_for(size_t total) {
  size_t g = (total + 255) / 256;
  if (g > 152 * 64) g = 152 * 64;
  if (g < 1) g = 1;
  return (int)g;
}

}  // namespace

// n_image: tokens of the embedding table (rows * row_len); t0 + nt must not
// exceed it
extern "C" int hkv_synth_image(void* q, void* k, void* v, int bf16, const float* pe,
                               const float* cq, unsigned long long seed, int S, int H, int D,
                               int C, int row_len, int n_image, int L, int l0, int nl, int t0,
                               int nt, float ks, float vs, cudaStream_t stream) {
  if (!q || !k || !v || !pe || !cq || S <= 0 || H <= 0 || D <= 0 || nl <= 0 || nt <= 0 ||
      l0 < 0 || l0 + nl > L || t0 < 0 || row_len <= 0 || t0 + nt > n_image)
    return 1;
  const size_t total = (size_t)nt * nl * S * H * D;
  synth_image_kernel<<<grid_for(total), 256, 0, stream>>>(q, k, v, bf16, pe, cq, seed, S, H, D,
                                                         C, row_len, L, l0, nl, t0, nt, ks, vs);
  return cudaGetLastError() == cudaSuccess ? 0 : 7;
}

extern "C" int hkv_synth_cond(void* kc, void* vc, int bf16, unsigned long long seed, int S,
                              int H, int D, int C, int l, float ks, float vs,
                              cudaStream_t stream) {
  if (!kc || !vc || S <= 0 || H <= 0 || D <= 0 || C < 0 || l < 0) return 1;
  if (C == 0) return 0;
  const size_t total = (size_t)S * H * C * D;
  synth_cond_kernel<<<grid_for(total), 256, 0, stream>>>(kc, vc, bf16, seed, S, H, D, C, l, ks,
                                                         vs);
  return cudaGetLastError() == cudaSuccess ? 0 : 7;
}
