// Inter-model junction of a Matryoshka suite (paper Eq. 1), forward and
// backward.  Per token, with o the output of sub-model m (D_m values) and e the
// fresh embedding of sub-model m+1 (D_{m+1} - D_m values):
//   o~ = o * ||e|| / ||o||   (0 when ||o|| = 0),   x = concat(o~, e)  or  concat(e, o~)
// Backward with g = dL/dx, s = ||e|| / ||o||:
//   dL/do = s (g_o - o (g_o . o) / ||o||^2)
//   dL/de = g_e + s (g_o . o) e / ||e||^2
// Both are row reductions followed by an elementwise pass, bound by HBM.  One
// warp owns a token, and each input byte is read from HBM once.  Three paths:
//   - register cache (rows whose segments need at most 8 vectors of 16 bytes
//     per lane): the warp issues every load of its row at once (o and e, and g
//     in the backward) and keeps them packed in registers, so a row costs one
//     memory latency;
//   - TMA ring (wider rows): persistent warps fetch whole rows into shared
//     memory with 1-D bulk copies, several rows ahead;
//   - streaming (rows too wide for two ring buffers): the row is read twice,
//     the second time from L2.
// Sums are fp32, accumulated per lane in column order, then across the warp,
// in every path, so all three give identical results.
#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

constexpr int kRowsPerBlock = 4;

// 16 bytes of E <-> N fp32 values.
template <typename E>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int N = 8;
  static __device__ __forceinline__ void unpack(const uint4& u, float (&f)[8]) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 h = *reinterpret_cast<const __nv_bfloat162*>(&w[i]);
      const float2 v = __bfloat1622float2(h);
      f[2 * i] = v.x;
      f[2 * i + 1] = v.y;
    }
  }
  static __device__ __forceinline__ uint4 pack(const float (&f)[8]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      __nv_bfloat162 h = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
      w[i] = *reinterpret_cast<uint32_t*>(&h);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
  }
};
template <>
struct Vec<float> {
  static constexpr int N = 4;
  static __device__ __forceinline__ void unpack(const uint4& u, float (&f)[4]) {
    f[0] = __uint_as_float(u.x);
    f[1] = __uint_as_float(u.y);
    f[2] = __uint_as_float(u.z);
    f[3] = __uint_as_float(u.w);
  }
  static __device__ __forceinline__ uint4 pack(const float (&f)[4]) {
    return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]),
                      __float_as_uint(f[3]));
  }
};

__device__ __forceinline__ uint4 ld16(const void* p) { return *reinterpret_cast<const uint4*>(p); }
__device__ __forceinline__ void st16(void* p, const uint4& v) { *reinterpret_cast<uint4*>(p) = v; }

// Tells the compiler the cached vectors may have changed, so it re-unpacks
// them after the reductions instead of keeping 8 floats per vector alive.
template <int R>
__device__ __forceinline__ void keep_packed(uint4 (&v)[R]) {
#pragma unroll
  for (int j = 0; j < R; ++j) asm volatile("" : "+r"(v[j].x), "+r"(v[j].y), "+r"(v[j].z), "+r"(v[j].w));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Lane `lane`'s vectors of a row segment of n elements: vector j holds
// elements (32 j + lane) N ... + N - 1; those past n read as zeros.
template <typename E, int R>
__device__ __forceinline__ void load_seg(const E* row, int n, int lane, uint4 (&v)[R]) {
  constexpr int N = Vec<E>::N;
#pragma unroll
  for (int j = 0; j < R; ++j) {
    const int k = (j * 32 + lane) * N;
    v[j] = k < n ? ld16(row + k) : make_uint4(0u, 0u, 0u, 0u);
  }
}

template <typename E, int R>
__device__ __forceinline__ float sumsq_cached(const uint4 (&v)[R]) {
  constexpr int N = Vec<E>::N;
  float acc = 0.f;
#pragma unroll
  for (int j = 0; j < R; ++j) {
    float f[N];
    Vec<E>::unpack(v[j], f);
#pragma unroll
    for (int i = 0; i < N; ++i) acc = fmaf(f[i], f[i], acc);
  }
  return acc;
}

template <typename E>
__device__ __forceinline__ float sumsq_stream(const E* row, int n, int lane) {
  constexpr int N = Vec<E>::N;
  float acc = 0.f;
  for (int k = lane * N; k < n; k += 32 * N) {
    float f[N];
    Vec<E>::unpack(ld16(row + k), f);
#pragma unroll
    for (int i = 0; i < N; ++i) acc = fmaf(f[i], f[i], acc);
  }
  return acc;
}

struct FwdRow {
  long long t;
  int de;
  const void *o, *e;
  void *xo, *xe;
};

template <typename E>
__device__ __forceinline__ FwdRow fwd_row(const JunctionParams& p, long long t) {
  const int de = p.d_next - p.d_prev;
  E* x = static_cast<E*>(p.x) + t * p.d_next;
  return {t, de, static_cast<const E*>(p.o) + t * p.d_prev, static_cast<const E*>(p.e) + t * de,
          x + (p.embed_first ? de : 0), x + (p.embed_first ? 0 : p.d_prev)};
}

// kR > 0: both segments fit kR cached vectors per lane; kR == 0: streaming.
template <typename E, int kR>
__global__ void __launch_bounds__(32 * kRowsPerBlock) junction_fwd_kernel(const JunctionParams p) {
  constexpr int N = Vec<E>::N;
  const long long t = static_cast<long long>(blockIdx.x) * kRowsPerBlock + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= p.T) return;
  const FwdRow r = fwd_row<E>(p, t);
  const E* o = static_cast<const E*>(r.o);
  const E* e = static_cast<const E*>(r.e);
  E* xo = static_cast<E*>(r.xo);
  E* xe = static_cast<E*>(r.xe);
  if constexpr (kR > 0) {
    uint4 vo[kR], ve[kR];
    load_seg<E, kR>(o, p.d_prev, lane, vo);
    load_seg<E, kR>(e, r.de, lane, ve);
    const float no = sqrtf(warp_sum(sumsq_cached<E, kR>(vo)));
    const float ne = sqrtf(warp_sum(sumsq_cached<E, kR>(ve)));
    const float s = no > 0.f ? ne / no : 0.f;
    keep_packed(vo);
#pragma unroll
    for (int j = 0; j < kR; ++j) {
      const int k = (j * 32 + lane) * N;
      if (k < p.d_prev) {
        float f[N];
        Vec<E>::unpack(vo[j], f);
#pragma unroll
        for (int i = 0; i < N; ++i) f[i] *= s;
        st16(xo + k, Vec<E>::pack(f));
      }
      if (k < r.de) st16(xe + k, ve[j]);
    }
  } else {
    const float no = sqrtf(warp_sum(sumsq_stream(o, p.d_prev, lane)));
    const float ne = sqrtf(warp_sum(sumsq_stream(e, r.de, lane)));
    const float s = no > 0.f ? ne / no : 0.f;
    for (int k = lane * N; k < p.d_prev; k += 32 * N) {
      float f[N];
      Vec<E>::unpack(ld16(o + k), f);
#pragma unroll
      for (int i = 0; i < N; ++i) f[i] *= s;
      st16(xo + k, Vec<E>::pack(f));
    }
    for (int k = lane * N; k < r.de; k += 32 * N) st16(xe + k, ld16(e + k));
  }
}

template <typename E, int kR>
__global__ void __launch_bounds__(32 * kRowsPerBlock) junction_bwd_kernel(const JunctionParams p) {
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
  float oo = 0.f, dot = 0.f, ee;
  if constexpr (kR > 0) {
    // Every input vector of the row is loaded at once and stays in registers.
    uint4 vo[kR], vg[kR], ve[kR], vge[kR];
    load_seg<E, kR>(o, p.d_prev, lane, vo);
    load_seg<E, kR>(go, p.d_prev, lane, vg);
    load_seg<E, kR>(e, de, lane, ve);
    load_seg<E, kR>(ge, de, lane, vge);
#pragma unroll
    for (int j = 0; j < kR; ++j) {
      float fo[N], fg[N];
      Vec<E>::unpack(vo[j], fo);
      Vec<E>::unpack(vg[j], fg);
#pragma unroll
      for (int i = 0; i < N; ++i) {
        oo = fmaf(fo[i], fo[i], oo);
        dot = fmaf(fg[i], fo[i], dot);
      }
    }
    oo = warp_sum(oo);
    dot = warp_sum(dot);
    ee = warp_sum(sumsq_cached<E, kR>(ve));
    const float no = sqrtf(oo), ne = sqrtf(ee);
    const float s = no > 0.f ? ne / no : 0.f;
    const float co = no > 0.f ? dot / oo : 0.f;                    // (g_o . o) / ||o||^2
    const float ce = (no > 0.f && ee > 0.f) ? s * dot / ee : 0.f;  // s (g_o . o) / ||e||^2
    keep_packed(vo);
    keep_packed(vg);
    keep_packed(ve);
#pragma unroll
    for (int j = 0; j < kR; ++j) {
      const int k = (j * 32 + lane) * N;
      if (k < p.d_prev) {
        float fo[N], fg[N], r[N];
        Vec<E>::unpack(vo[j], fo);
        Vec<E>::unpack(vg[j], fg);
#pragma unroll
        for (int i = 0; i < N; ++i) r[i] = s * fmaf(-fo[i], co, fg[i]);
        st16(d_o + k, Vec<E>::pack(r));
      }
      if (k < de) {
        float fe[N], fg[N], r[N];
        Vec<E>::unpack(ve[j], fe);
        Vec<E>::unpack(vge[j], fg);
#pragma unroll
        for (int i = 0; i < N; ++i) r[i] = fmaf(ce, fe[i], fg[i]);
        st16(d_e + k, Vec<E>::pack(r));
      }
    }
  } else {
    for (int k = lane * N; k < p.d_prev; k += 32 * N) {
      float fo[N], fg[N];
      Vec<E>::unpack(ld16(o + k), fo);
      Vec<E>::unpack(ld16(go + k), fg);
#pragma unroll
      for (int i = 0; i < N; ++i) {
        oo = fmaf(fo[i], fo[i], oo);
        dot = fmaf(fg[i], fo[i], dot);
      }
    }
    oo = warp_sum(oo);
    dot = warp_sum(dot);
    ee = warp_sum(sumsq_stream(e, de, lane));
    const float no = sqrtf(oo), ne = sqrtf(ee);
    const float s = no > 0.f ? ne / no : 0.f;
    const float co = no > 0.f ? dot / oo : 0.f;
    const float ce = (no > 0.f && ee > 0.f) ? s * dot / ee : 0.f;
    for (int k = lane * N; k < p.d_prev; k += 32 * N) {
      float fo[N], fg[N], r[N];
      Vec<E>::unpack(ld16(o + k), fo);
      Vec<E>::unpack(ld16(go + k), fg);
#pragma unroll
      for (int i = 0; i < N; ++i) r[i] = s * fmaf(-fo[i], co, fg[i]);
      st16(d_o + k, Vec<E>::pack(r));
    }
    for (int k = lane * N; k < de; k += 32 * N) {
      float fe[N], fg[N], r[N];
      Vec<E>::unpack(ld16(e + k), fe);
      Vec<E>::unpack(ld16(ge + k), fg);
#pragma unroll
      for (int i = 0; i < N; ++i) r[i] = fmaf(ce, fe[i], fg[i]);
      st16(d_e + k, Vec<E>::pack(r));
    }
  }
}

// ---------------------------------------------------------------- TMA ring
// Rows wider than the register cache.  Persistent CTAs of `warps` warps; each
// warp owns a ring of `stages` row buffers in shared memory and the rows gw,
// gw + GW, ... (gw its global warp index, GW the warps of the grid).  Its lane
// 0 fetches whole rows (o and e, and g in the backward) with 1-D bulk copies
// that complete on the buffer's mbarrier, `stages` rows ahead, so every SM
// keeps several rows of HBM reads in flight whatever T is.  The warp computes
// a row from shared memory, in the same lane and column order as the kernels
// above, and stores its outputs with coalesced 16-byte stores.
constexpr int kRingWarps = 4;
constexpr int kRingStages = 4;
constexpr uint32_t kRingSmem = 220 * 1024;  // dynamic shared memory a CTA may use
constexpr uint64_t kDrainNs = 100000000ull;

template <typename E>
__device__ __forceinline__ uint4 ld16s(const E* p) { return *reinterpret_cast<const uint4*>(p); }

template <typename E, bool kBwd>
__global__ void __launch_bounds__(32 * kRingWarps)
    junction_ring_kernel(const JunctionParams p, int stages, uint32_t stage_bytes) {
  constexpr int N = Vec<E>::N;
  extern __shared__ __align__(128) uint8_t ring_smem[];
  __shared__ __align__(8) uint64_t bars[kRingWarps * kRingStages];
  __shared__ int abort_flag;
  const int nw = static_cast<int>(blockDim.x >> 5), w = static_cast<int>(threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const long long GW = static_cast<long long>(gridDim.x) * nw;
  const long long gw = static_cast<long long>(blockIdx.x) * nw + w;
  const int de = p.d_next - p.d_prev;
  const uint32_t ob = p.d_prev * sizeof(E), eb = de * sizeof(E);
  const uint32_t gb = kBwd ? p.d_next * sizeof(E) : 0u;
  uint8_t* ring = ring_smem + static_cast<size_t>(w) * stages * stage_bytes;
  const uint32_t ring_s = smem_u32(ring), bar0 = smem_u32(&bars[w * kRingStages]);
  if (threadIdx.x == 0) abort_flag = 0;
  if (lane == 0)
    for (int st = 0; st < stages; ++st) mbar_init(bar0 + 8u * st, 1);
  fence_barrier_init();
  __syncthreads();
  const E* o = static_cast<const E*>(p.o);
  const E* e = static_cast<const E*>(p.e);
  const E* g = static_cast<const E*>(p.g);
  auto fetch = [&](long long r, int st) {
    const uint32_t dst = ring_s + static_cast<uint32_t>(st) * stage_bytes, bar = bar0 + 8u * st;
    mbar_arrive_expect_tx(bar, ob + eb + gb);
    bulk_load_1d(dst, o + r * p.d_prev, ob, bar);
    bulk_load_1d(dst + ob, e + r * de, eb, bar);
    if (kBwd) bulk_load_1d(dst + ob + eb, g + r * p.d_next, gb, bar);
  };
  if (lane == 0)
    for (int st = 0; st < stages; ++st)
      if (gw + st * GW < p.T) fetch(gw + st * GW, st);
  long long i = 0;
  bool ok = true;
  for (long long r = gw; r < p.T; r += GW, ++i) {
    const int st = static_cast<int>(i % stages);
    // Every lane waits, but the warp leaves together: a lane that saw the
    // buffer land must not go on to the full-warp reductions below while a
    // lane that saw another warp's abort has left.
    const bool landed =
        mbar_wait(bar0 + 8u * st, static_cast<uint32_t>((i / stages) & 1), &abort_flag, p.status);
    if (!__all_sync(0xffffffffu, landed)) {
      ok = false;
      break;
    }
    const E* os = reinterpret_cast<const E*>(ring + static_cast<size_t>(st) * stage_bytes);
    const E* es = os + p.d_prev;
    if constexpr (!kBwd) {
      float so = 0.f, se = 0.f;
      for (int k = lane * N; k < p.d_prev; k += 32 * N) {
        float f[N];
        Vec<E>::unpack(ld16s(os + k), f);
#pragma unroll
        for (int q = 0; q < N; ++q) so = fmaf(f[q], f[q], so);
      }
      for (int k = lane * N; k < de; k += 32 * N) {
        float f[N];
        Vec<E>::unpack(ld16s(es + k), f);
#pragma unroll
        for (int q = 0; q < N; ++q) se = fmaf(f[q], f[q], se);
      }
      const float no = sqrtf(warp_sum(so)), ne = sqrtf(warp_sum(se));
      const float sc = no > 0.f ? ne / no : 0.f;
      E* x = static_cast<E*>(p.x) + r * p.d_next;
      E* xo = x + (p.embed_first ? de : 0);
      E* xe = x + (p.embed_first ? 0 : p.d_prev);
      for (int k = lane * N; k < p.d_prev; k += 32 * N) {
        float f[N];
        Vec<E>::unpack(ld16s(os + k), f);
#pragma unroll
        for (int q = 0; q < N; ++q) f[q] *= sc;
        st16(xo + k, Vec<E>::pack(f));
      }
      for (int k = lane * N; k < de; k += 32 * N) st16(xe + k, ld16s(es + k));
    } else {
      const E* gs = es + de;
      const E* gos = gs + (p.embed_first ? de : 0);
      const E* ges = gs + (p.embed_first ? 0 : p.d_prev);
      float oo = 0.f, dot = 0.f, ee = 0.f;
      for (int k = lane * N; k < p.d_prev; k += 32 * N) {
        float fo[N], fg[N];
        Vec<E>::unpack(ld16s(os + k), fo);
        Vec<E>::unpack(ld16s(gos + k), fg);
#pragma unroll
        for (int q = 0; q < N; ++q) {
          oo = fmaf(fo[q], fo[q], oo);
          dot = fmaf(fg[q], fo[q], dot);
        }
      }
      for (int k = lane * N; k < de; k += 32 * N) {
        float f[N];
        Vec<E>::unpack(ld16s(es + k), f);
#pragma unroll
        for (int q = 0; q < N; ++q) ee = fmaf(f[q], f[q], ee);
      }
      oo = warp_sum(oo);
      dot = warp_sum(dot);
      ee = warp_sum(ee);
      const float no = sqrtf(oo), ne = sqrtf(ee);
      const float sc = no > 0.f ? ne / no : 0.f;
      const float co = no > 0.f ? dot / oo : 0.f;                     // (g_o . o) / ||o||^2
      const float ce = (no > 0.f && ee > 0.f) ? sc * dot / ee : 0.f;  // s (g_o . o) / ||e||^2
      E* d_o = static_cast<E*>(p.d_o) + r * p.d_prev;
      E* d_e = static_cast<E*>(p.d_e) + r * de;
      for (int k = lane * N; k < p.d_prev; k += 32 * N) {
        float fo[N], fg[N], y[N];
        Vec<E>::unpack(ld16s(os + k), fo);
        Vec<E>::unpack(ld16s(gos + k), fg);
#pragma unroll
        for (int q = 0; q < N; ++q) y[q] = sc * fmaf(-fo[q], co, fg[q]);
        st16(d_o + k, Vec<E>::pack(y));
      }
      for (int k = lane * N; k < de; k += 32 * N) {
        float fe[N], fg[N], y[N];
        Vec<E>::unpack(ld16s(es + k), fe);
        Vec<E>::unpack(ld16s(ges + k), fg);
#pragma unroll
        for (int q = 0; q < N; ++q) y[q] = fmaf(ce, fe[q], fg[q]);
        st16(d_e + k, Vec<E>::pack(y));
      }
    }
    // Every lane's reads of this buffer precede the copy that refills it.
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0 && r + stages * GW < p.T) fetch(r + stages * GW, st);
  }
  if (!ok && lane == 0) {
    // The copies already issued (iterations i .. i + stages - 1) must land
    // before this CTA's shared memory goes away.
    for (long long k = i; k < i + stages; ++k)
      if (gw + k * GW < p.T)
        mbar_wait_drain(bar0 + 8u * static_cast<uint32_t>(k % stages),
                        static_cast<uint32_t>((k / stages) & 1), kDrainNs, p.status);
  }
}

// Ring shape for a row of `row_bytes`: 4 warps per CTA with 2 to 4 buffers
// each, two CTAs per SM when they fit, else one.  Returns false for rows too
// wide for that (over 27.5 KB), which stream instead: fewer than four warps
// per SM cannot keep HBM busy.  (Eight warps per CTA measured no faster.)
bool ring_shape(uint32_t row_bytes, int& warps, int& stages) {
  for (const int ctas : {2, 1}) {
    const long long st = kRingSmem / (static_cast<long long>(ctas) * kRingWarps * row_bytes);
    if (st >= 2) {
      warps = kRingWarps;
      stages = st > kRingStages ? kRingStages : static_cast<int>(st);
      return true;
    }
  }
  return false;
}

template <typename E, bool kBwd>
cudaError_t ring_launch(const JunctionParams& p, cudaStream_t s, bool& launched) {
  launched = false;
  const uint32_t elt = sizeof(E);
  const uint32_t row = (static_cast<uint32_t>(p.d_next) + (kBwd ? p.d_next : 0)) * elt;
  int warps = 0, stages = 0;
  if (!ring_shape(row, warps, stages)) return cudaSuccess;
  const size_t smem = static_cast<size_t>(warps) * stages * row;
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
      &per_sm, junction_ring_kernel<E, kBwd>, 32 * warps, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaSuccess;
  const long long need = (p.T + warps - 1) / warps;
  const long long most = static_cast<long long>(p.sms > 0 ? p.sms : 1) * per_sm;
  const unsigned blocks = static_cast<unsigned>(need < most ? need : most);
  junction_ring_kernel<E, kBwd><<<blocks, 32 * warps, smem, s>>>(p, stages, row);
  launched = true;
  return cudaGetLastError();
}

// Cached vectors per lane for a row whose segments are d_prev and d_next -
// d_prev elements of `elt` bytes: the smallest of 1, 2, 4, 8 that holds both,
// or 0 when a segment needs more.  At 12 vectors the backward needed 254
// registers and ran ~10% slower than the TMA ring.
int cache_vectors(int d_prev, int d_next, int elt) {
  const int per = 32 * (16 / elt);  // elements per cached vector across the warp
  const int need_o = (d_prev + per - 1) / per, need_e = (d_next - d_prev + per - 1) / per;
  const int need = need_o > need_e ? need_o : need_e;
  for (const int r : {1, 2, 4, 8})
    if (need <= r) return r;
  return 0;
}

template <typename E>
cudaError_t fwd_launch(const JunctionParams& p, int r, unsigned blocks, cudaStream_t s) {
  const dim3 b(32 * kRowsPerBlock);
  switch (r) {
    case 1: junction_fwd_kernel<E, 1><<<blocks, b, 0, s>>>(p); break;
    case 2: junction_fwd_kernel<E, 2><<<blocks, b, 0, s>>>(p); break;
    case 4: junction_fwd_kernel<E, 4><<<blocks, b, 0, s>>>(p); break;
    case 8: junction_fwd_kernel<E, 8><<<blocks, b, 0, s>>>(p); break;
    default: junction_fwd_kernel<E, 0><<<blocks, b, 0, s>>>(p); break;
  }
  return cudaGetLastError();
}

template <typename E>
cudaError_t bwd_launch(const JunctionParams& p, int r, unsigned blocks, cudaStream_t s) {
  const dim3 b(32 * kRowsPerBlock);
  switch (r) {
    case 1: junction_bwd_kernel<E, 1><<<blocks, b, 0, s>>>(p); break;
    case 2: junction_bwd_kernel<E, 2><<<blocks, b, 0, s>>>(p); break;
    case 4: junction_bwd_kernel<E, 4><<<blocks, b, 0, s>>>(p); break;
    case 8: junction_bwd_kernel<E, 8><<<blocks, b, 0, s>>>(p); break;
    default: junction_bwd_kernel<E, 0><<<blocks, b, 0, s>>>(p); break;
  }
  return cudaGetLastError();
}

}  // namespace

// Register cache when a row fits 8 vectors per lane, else the TMA ring, else
// (rows too wide for two ring buffers) the streaming kernel.
cudaError_t launch_junction_fwd(const JunctionParams& p, bool fp32, cudaStream_t s) {
  const long long blocks = (p.T + kRowsPerBlock - 1) / kRowsPerBlock;
  if (blocks <= 0) return cudaSuccess;
  const int r = cache_vectors(p.d_prev, p.d_next, fp32 ? 4 : 2);
  if (r == 0) {
    bool launched = false;
    const cudaError_t e = fp32 ? ring_launch<float, false>(p, s, launched)
                               : ring_launch<__nv_bfloat16, false>(p, s, launched);
    if (e != cudaSuccess || launched) return e;
  }
  return fp32 ? fwd_launch<float>(p, r, static_cast<unsigned>(blocks), s)
              : fwd_launch<__nv_bfloat16>(p, r, static_cast<unsigned>(blocks), s);
}

cudaError_t launch_junction_bwd(const JunctionParams& p, bool fp32, cudaStream_t s) {
  const long long blocks = (p.T + kRowsPerBlock - 1) / kRowsPerBlock;
  if (blocks <= 0) return cudaSuccess;
  const int r = cache_vectors(p.d_prev, p.d_next, fp32 ? 4 : 2);
  if (r == 0) {
    bool launched = false;
    const cudaError_t e = fp32 ? ring_launch<float, true>(p, s, launched)
                               : ring_launch<__nv_bfloat16, true>(p, s, launched);
    if (e != cudaSuccess || launched) return e;
  }
  return fp32 ? bwd_launch<float>(p, r, static_cast<unsigned>(blocks), s)
              : bwd_launch<__nv_bfloat16>(p, r, static_cast<unsigned>(blocks), s);
}

cudaError_t setup_junction_kernels() {
  cudaError_t e;
#define MLS_SET(E, B)                                                                        \
  e = cudaFuncSetAttribute(junction_ring_kernel<E, B>,                                       \
                           cudaFuncAttributeMaxDynamicSharedMemorySize, kRingSmem);          \
  if (e != cudaSuccess) return e;
  MLS_SET(float, false)
  MLS_SET(float, true)
  MLS_SET(__nv_bfloat16, false)
  MLS_SET(__nv_bfloat16, true)
#undef MLS_SET
  return cudaSuccess;
}

}  // namespace mls
