// Inter-model junction of a Matryoshka suite (paper Eq. 1), forward and
// backward.  Per token, with o the output of sub-model m (D_m values) and e the
// fresh embedding of sub-model m+1 (D_{m+1} - D_m values):
//   o~ = o * ||e|| / ||o||   (0 when ||o|| = 0),   x = concat(o~, e)  or  concat(e, o~)
// Backward with g = dL/dx, s = ||e|| / ||o||:
//   dL/do = s (g_o - o (g_o . o) / ||o||^2)
//   dL/de = g_e + s (g_o . o) e / ||e||^2
// Both are row reductions plus an elementwise pass, bound by HBM: one warp per
// token, 16-byte vector accesses, fp32 sums; the second pass re-reads the row
// from L1/L2.
#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

constexpr int kRowsPerBlock = 8;

template <typename E>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int N = 8;
  static __device__ __forceinline__ void load(const void* p, float (&f)[8]) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 h = *reinterpret_cast<const __nv_bfloat162*>(&w[i]);
      const float2 v = __bfloat1622float2(h);
      f[2 * i] = v.x;
      f[2 * i + 1] = v.y;
    }
  }
  static __device__ __forceinline__ void store(void* p, const float (&f)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
      w[i] = *reinterpret_cast<uint32_t*>(&h);
    }
    *reinterpret_cast<uint4*>(p) = make_uint4(w[0], w[1], w[2], w[3]);
  }
};
template <>
struct Vec<float> {
  static constexpr int N = 4;
  static __device__ __forceinline__ void load(const void* p, float (&f)[4]) {
    const float4 v = *reinterpret_cast<const float4*>(p);
    f[0] = v.x;
    f[1] = v.y;
    f[2] = v.z;
    f[3] = v.w;
  }
  static __device__ __forceinline__ void store(void* p, const float (&f)[4]) {
    *reinterpret_cast<float4*>(p) = make_float4(f[0], f[1], f[2], f[3]);
  }
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename E>
__device__ __forceinline__ float sumsq(const E* row, int n, int lane) {
  constexpr int N = Vec<E>::N;
  float acc = 0.f;
  for (int k = lane * N; k < n; k += 32 * N) {
    float f[N];
    Vec<E>::load(row + k, f);
#pragma unroll
    for (int i = 0; i < N; ++i) acc = fmaf(f[i], f[i], acc);
  }
  return warp_sum(acc);
}

template <typename E>
__global__ void __launch_bounds__(32 * kRowsPerBlock)
    junction_fwd_kernel(const JunctionParams p) {
  constexpr int N = Vec<E>::N;
  const long long t = static_cast<long long>(blockIdx.x) * kRowsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= p.T) return;
  const int de = p.d_next - p.d_prev;
  const E* o = static_cast<const E*>(p.o) + t * p.d_prev;
  const E* e = static_cast<const E*>(p.e) + t * de;
  E* x = static_cast<E*>(p.x) + t * p.d_next;
  const float no = sqrtf(sumsq(o, p.d_prev, lane));
  const float ne = sqrtf(sumsq(e, de, lane));
  const float s = no > 0.f ? ne / no : 0.f;
  E* xo = x + (p.embed_first ? de : 0);
  E* xe = x + (p.embed_first ? 0 : p.d_prev);
  for (int k = lane * N; k < p.d_prev; k += 32 * N) {
    float f[N];
    Vec<E>::load(o + k, f);
#pragma unroll
    for (int i = 0; i < N; ++i) f[i] *= s;
    Vec<E>::store(xo + k, f);
  }
  for (int k = lane * N; k < de; k += 32 * N) {
    float f[N];
    Vec<E>::load(e + k, f);
    Vec<E>::store(xe + k, f);
  }
}

template <typename E>
__global__ void __launch_bounds__(32 * kRowsPerBlock)
    junction_bwd_kernel(const JunctionParams p) {
  constexpr int N = Vec<E>::N;
  const long long t = static_cast<long long>(blockIdx.x) * kRowsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= p.T) return;
  const int de = p.d_next - p.d_prev;
  const E* o = static_cast<const E*>(p.o) + t * p.d_prev;
  const E* e = static_cast<const E*>(p.e) + t * de;
  const E* g = static_cast<const E*>(p.g) + t * p.d_next;
  const E* go = g + (p.embed_first ? de : 0);
  const E* ge = g + (p.embed_first ? 0 : p.d_prev);
  E* d_o = static_cast<E*>(p.d_o) + t * p.d_prev;
  E* d_e = static_cast<E*>(p.d_e) + t * de;
  float oo = 0.f, dot = 0.f;
  for (int k = lane * N; k < p.d_prev; k += 32 * N) {
    float fo[N], fg[N];
    Vec<E>::load(o + k, fo);
    Vec<E>::load(go + k, fg);
#pragma unroll
    for (int i = 0; i < N; ++i) {
      oo = fmaf(fo[i], fo[i], oo);
      dot = fmaf(fg[i], fo[i], dot);
    }
  }
  oo = warp_sum(oo);
  dot = warp_sum(dot);
  const float ee = sumsq(e, de, lane);
  const float no = sqrtf(oo), ne = sqrtf(ee);
  const float s = no > 0.f ? ne / no : 0.f;
  const float co = no > 0.f ? dot / oo : 0.f;             // (g_o . o) / ||o||^2
  const float ce = (no > 0.f && ee > 0.f) ? s * dot / ee : 0.f;  // s (g_o . o) / ||e||^2
  for (int k = lane * N; k < p.d_prev; k += 32 * N) {
    float fo[N], fg[N], r[N];
    Vec<E>::load(o + k, fo);
    Vec<E>::load(go + k, fg);
#pragma unroll
    for (int i = 0; i < N; ++i) r[i] = s * fmaf(-fo[i], co, fg[i]);
    Vec<E>::store(d_o + k, r);
  }
  for (int k = lane * N; k < de; k += 32 * N) {
    float fe[N], fg[N], r[N];
    Vec<E>::load(e + k, fe);
    Vec<E>::load(ge + k, fg);
#pragma unroll
    for (int i = 0; i < N; ++i) r[i] = fmaf(ce, fe[i], fg[i]);
    Vec<E>::store(d_e + k, r);
  }
}

}  // namespace

cudaError_t launch_junction_fwd(const JunctionParams& p, bool fp32, cudaStream_t s) {
  const long long blocks = (p.T + kRowsPerBlock - 1) / kRowsPerBlock;
  if (blocks <= 0) return cudaSuccess;
  if (fp32)
    junction_fwd_kernel<float><<<static_cast<unsigned>(blocks), 32 * kRowsPerBlock, 0, s>>>(p);
  else
    junction_fwd_kernel<__nv_bfloat16><<<static_cast<unsigned>(blocks), 32 * kRowsPerBlock, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_junction_bwd(const JunctionParams& p, bool fp32, cudaStream_t s) {
  const long long blocks = (p.T + kRowsPerBlock - 1) / kRowsPerBlock;
  if (blocks <= 0) return cudaSuccess;
  if (fp32)
    junction_bwd_kernel<float><<<static_cast<unsigned>(blocks), 32 * kRowsPerBlock, 0, s>>>(p);
  else
    junction_bwd_kernel<__nv_bfloat16><<<static_cast<unsigned>(blocks), 32 * kRowsPerBlock, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace mls
