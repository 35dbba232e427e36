// Speculative-decoding verify step for a nested draft / verifier pair (paper
// Sec. 2 "Speculative Decoding"; Sec. 3.2.3 samples with temperature 0.4 and
// nucleus p = 0.9, or greedily), standard speculative sampling:
//   x_i is accepted iff q_i(x_i) > 0 and u_i * q_i(x_i) < p_i(x_i);
//   at the first rejection k, the next token is sampled from
//   norm(max(0, p_k - q_k)) (from p_k if that is all zero); if all gamma are
//   accepted it is sampled from p_gamma;  sample(r, u) = the smallest v with
//   sum_{w <= v} r_w > u * sum_w r_w.
// p and q are nucleus(softmax(z / temperature)): tokens ordered by
// probability (then by index) are kept through the first one at which the
// cumulative probability reaches top_p, then renormalised.  Greedy: accept
// while x_i == argmax of the verifier's logits (lowest index on ties).
//
// The logits GEMM's epilogue (mls_gemm.cu) leaves, per row and column tile t
// of 256, e_t[v] = 2^((z[v] - m_t) log2(e) / T) and (m_t, sum_t), or for greedy
// only (m_t, argmax_t).  Here, with m = max_t m_t and f_t = 2^((m_t - m) log2(e)/T),
// every token's unnormalised probability is e[v] = e_t[v] f_t (<= 1) and
// S = sum_t sum_t f_t:
//   spec_row_kernel (one CTA per row, sampling only) finds the row's nucleus:
//     the boundary value b = the largest e with mass(e' >= b) >= top_p S, by
//     bisection over the bit patterns of e (non-negative floats order like
//     their bits).  The first pass splits at 2^-8 of the maximum and keeps the
//     few tokens above it in shared memory; later passes narrow the bracket,
//     compacting survivors into shared memory once they fit, and the last
//     <= 256 are resolved exactly.  Then the c lowest-index tokens with e == b
//     that the cumulative needs.
//   spec_sample_kernel (one CTA per sequence) decides acceptance of every
//     drafted token from the rows' nucleus states, takes the first rejection
//     and samples by inverse CDF in index order; for greedy it reduces the
//     tile argmaxes.
// Every reduction has a fixed order, so a call is deterministic.
#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kStep = 128;              // elements one warp covers per float4 step
constexpr int kUnroll = 6;              // independent float4 loads in flight per lane
constexpr int kFinish = 256;            // candidates resolved exactly
constexpr uint32_t kOneKey = 0x3f800000u;     // bit pattern of 1.0f
constexpr uint32_t kFirstMid = 0x3b800000u;   // 2^-8
constexpr uint32_t kSecondMid = 0x37800000u;  // 2^-16
static_assert(kFinish <= kThreads, "one candidate per thread in the exact finish");

// Per-warp partials of a block reduction (f, n, k) and the combined results
// (rf, rn, rk) that warp 0 writes for everyone.
template <int NW>
struct SharedT {
  float f[NW][2];
  int n[NW][3];
  uint32_t k[NW][4];
  int wbase[NW];
  int wcnt[NW];
  float rf[2];
  int rn[3];
  uint32_t rk[4];
};
using Shared = SharedT<kWarps>;
constexpr int kSampleWarps = 32;  // the per-sequence sampler runs 1024 threads

__device__ __forceinline__ int lane_id() { return threadIdx.x & 31; }
__device__ __forceinline__ int warp_id() { return threadIdx.x >> 5; }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ int warp_incl_scan(int v) {
  const int l = lane_id();
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, v, o);
    if (l >= o) v += t;
  }
  return v;
}

__device__ __forceinline__ float warp_incl_scan(float v) {
  const int l = lane_id();
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float t = __shfl_up_sync(0xffffffffu, v, o);
    if (l >= o) v += t;
  }
  return v;
}

__device__ __forceinline__ float comp(const float4& v, int j) {
  return j == 0 ? v.x : j == 1 ? v.y : j == 2 ? v.z : v.w;
}

// Block reductions: each warp reduces by a butterfly, lane 0 parks the
// warp's partial, warp 0 combines the 16 partials by a butterfly and parks the
// result for every thread.  Fixed order throughout.
__device__ __forceinline__ void argmax_step(float& v, int& idx, float ov, int oi) {
  if (ov > v || (ov == v && oi < idx)) {
    v = ov;
    idx = oi;
  }
}

// (max value, lowest index attaining it).
template <int NW>
__device__ void block_argmax(float& v, int& idx, SharedT<NW>& sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
    argmax_step(v, idx, __shfl_xor_sync(0xffffffffu, v, o), __shfl_xor_sync(0xffffffffu, idx, o));
  __syncthreads();
  if (lane_id() == 0) {
    sh.f[warp_id()][0] = v;
    sh.n[warp_id()][0] = idx;
  }
  __syncthreads();
  if (warp_id() == 0) {
    const int l = lane_id();
    float wv = l < NW ? sh.f[l][0] : -INFINITY;
    int wi = l < NW ? sh.n[l][0] : 0x7fffffff;
#pragma unroll
    for (int o = NW / 2; o > 0; o >>= 1)
      argmax_step(wv, wi, __shfl_xor_sync(0xffffffffu, wv, o), __shfl_xor_sync(0xffffffffu, wi, o));
    if (l == 0) {
      sh.rf[0] = wv;
      sh.rn[0] = wi;
    }
  }
  __syncthreads();
  v = sh.rf[0];
  idx = sh.rn[0];
}

// Sums of a float and an int.
template <int NW>
__device__ void block_sum2(float& f, int& n, SharedT<NW>& sh) {
  f = warp_sum(f);
  n = static_cast<int>(__reduce_add_sync(0xffffffffu, static_cast<unsigned>(n)));
  __syncthreads();
  if (lane_id() == 0) {
    sh.f[warp_id()][0] = f;
    sh.n[warp_id()][0] = n;
  }
  __syncthreads();
  if (warp_id() == 0) {
    const int l = lane_id();
    float wf = l < NW ? sh.f[l][0] : 0.f;
    int wn = l < NW ? sh.n[l][0] : 0;
#pragma unroll
    for (int o = NW / 2; o > 0; o >>= 1) {
      wf += __shfl_xor_sync(0xffffffffu, wf, o);
      wn += __shfl_xor_sync(0xffffffffu, wn, o);
    }
    if (l == 0) {
      sh.rf[0] = wf;
      sh.rn[0] = wn;
    }
  }
  __syncthreads();
  f = sh.rf[0];
  n = sh.rn[0];
}

template <int NW>
__device__ uint32_t block_max_u(uint32_t v, SharedT<NW>& sh) {
  v = __reduce_max_sync(0xffffffffu, v);
  __syncthreads();
  if (lane_id() == 0) sh.k[warp_id()][0] = v;
  __syncthreads();
  if (warp_id() == 0) {
    const uint32_t w = __reduce_max_sync(0xffffffffu, lane_id() < NW ? sh.k[lane_id()][0] : 0u);
    if (lane_id() == 0) sh.rk[0] = w;
  }
  __syncthreads();
  return sh.rk[0];
}

// Per-row softmax statistics from the per-tile ones: m, S and f_t (into the
// shared table and, if fg is not null, into global memory).
__device__ void row_stats(const float* st, int tiles, float scale, float* ftab, float* fg,
                          float& m, float& S, Shared& sh) {
  float mv = -INFINITY;
  int unused = 0;
  for (int t = threadIdx.x; t < tiles; t += kThreads) mv = fmaxf(mv, st[2 * t]);
  block_argmax(mv, unused, sh);
  m = mv;
  float s = 0.f;
  for (int t = threadIdx.x; t < tiles; t += kThreads) {
    const float f = fast_exp2((st[2 * t] - m) * scale);
    ftab[t] = f;
    if (fg) fg[t] = f;
    s = fmaf(st[2 * t + 1], f, s);
  }
  block_sum2(s, unused, sh);  // its barriers also publish ftab
  S = s;
}

// Visits a row of unnormalised probabilities e[v] = e_t[v] f_t, warp w taking
// the 128-element steps w, w + 16, ... (kUnroll of them per iteration):
// `f(i0, e4, V)` gets the lane's 4 consecutive elements from index i0 (those
// at or past V are not meaningful).  The loop is warp-uniform, so f may use
// warp collectives.  Rows are 16-byte aligned and padded to 4 elements.
template <int NW, typename F>
__device__ __forceinline__ void for_row(const float* et, const float* ftab, long long V, F&& f) {
  const int l = lane_id();
  constexpr long long kStride = static_cast<long long>(NW) * kStep;
  for (long long base = static_cast<long long>(warp_id()) * kStep; base < V;
       base += kUnroll * kStride) {
    float4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const long long i0 = base + u * kStride + l * 4;
      v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (i0 < V) v[u] = __ldg(reinterpret_cast<const float4*>(et + i0));
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const long long i0 = base + u * kStride + l * 4;
      if (i0 < V) {
        const float fm = ftab[i0 / kGemmBN];
        v[u].x *= fm;
        v[u].y *= fm;
        v[u].z *= fm;
        v[u].w *= fm;
      }
      f(i0, v[u], V);
    }
  }
}

// Statistics of one bisection pass over the candidates with key in [lo, hi),
// split at mid.  With d = key - lo (unsigned), mo = mid - lo, w = hi - lo and
// wm = w - mo: the lower side is d < mo, the upper side d - mo < wm.  Kept:
// mass and count of the upper side, count of the lower side and, when
// tracked, the smallest and largest key on each side.
struct PassStats {
  float mass_ge = 0.f;
  int cnt_ge = 0, cnt_lt = 0;
  uint32_t min_ge = 0xffffffffu, max_ge = 0u, min_lt = 0xffffffffu, max_lt = 0u;
  template <bool kTrack>
  __device__ __forceinline__ void add(float e, uint32_t lo, uint32_t mo, uint32_t wm) {
    const uint32_t key = __float_as_uint(e);
    const uint32_t d = key - lo;
    const bool lt = d < mo, ge = d - mo < wm;
    cnt_lt += lt;
    cnt_ge += ge;
    mass_ge += ge ? e : 0.f;
    if (kTrack) {
      if (lt) {
        min_lt = min(min_lt, key);
        max_lt = max(max_lt, key);
      }
      if (ge) {
        min_ge = min(min_ge, key);
        max_ge = max(max_ge, key);
      }
    }
  }
};

// One bisection pass over a whole row (e = e_t f_t), warps taking 128-token
// steps w, w + 16, ..., kUnroll steps per iteration; only the row's last
// float4 can be partial.
template <bool kTrack>
__device__ __forceinline__ void row_pass(const float* et, const float* ftab, int V, uint32_t lo,
                                         uint32_t mo, uint32_t wm, PassStats& ps) {
  const int l = lane_id();
  constexpr int kStride = kWarps * kStep;
  for (int base = warp_id() * kStep; base < V; base += kUnroll * kStride) {
    float4 v[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int s0 = base + u * kStride, i0 = s0 + l * 4;
      // a tile whose maximum lies below the bracket holds no candidate
      const bool live = s0 < V && __float_as_uint(ftab[static_cast<unsigned>(s0) / kGemmBN]) >= lo;
      v[u] = live && i0 < V ? __ldg(reinterpret_cast<const float4*>(et + i0))
                            : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int i0 = base + u * kStride + l * 4;
      if (i0 < V) {
        const float fm = ftab[static_cast<unsigned>(i0) / kGemmBN];
        if (__float_as_uint(fm) < lo) continue;
        const float e0 = v[u].x * fm, e1 = v[u].y * fm, e2 = v[u].z * fm, e3 = v[u].w * fm;
        ps.add<kTrack>(e0, lo, mo, wm);
        if (i0 + 4 <= V) {
          ps.add<kTrack>(e1, lo, mo, wm);
          ps.add<kTrack>(e2, lo, mo, wm);
          ps.add<kTrack>(e3, lo, mo, wm);
        } else {
          if (i0 + 1 < V) ps.add<kTrack>(e1, lo, mo, wm);
          if (i0 + 2 < V) ps.add<kTrack>(e2, lo, mo, wm);
        }
      }
    }
  }
}

// The column tiles whose factor f_t has a key of at least min_key (so the
// only tiles that can hold an e >= that value, since every e of tile t is at
// most f_t), in tile order, into kept[]; returns their number.  Needs ftab
// published; the trailing barrier publishes kept[].
template <int NW>
__device__ int kept_tiles(const float* ftab, int tiles, uint32_t min_key, int* kept,
                          SharedT<NW>& sh) {
  int nk = 0;
  for (int c0 = 0; c0 < tiles; c0 += NW * 32) {
    const int t = c0 + static_cast<int>(threadIdx.x);
    const bool keep = t < tiles && __float_as_uint(ftab[t]) >= min_key;
    const unsigned bal = __ballot_sync(0xffffffffu, keep);
    if (lane_id() == 0) sh.wcnt[warp_id()] = __popc(bal);
    __syncthreads();
    int at = nk, total = 0;
    for (int w = 0; w < NW; ++w) {
      const int c = sh.wcnt[w];
      if (w < warp_id()) at += c;
      total += c;
    }
    if (keep) kept[at + __popc(bal & ((1u << lane_id()) - 1u))] = t;
    nk += total;
    __syncthreads();  // sh.wcnt is rewritten next
  }
  return nk;
}

// The first bisection pass over a row: the split at 2^-8 of the maximum.
// Only the kept tiles are read.  Warp w takes kept[w], kept[w + kWarps], ...,
// kFirstTiles of them per round with all their loads in flight, so a peaked
// row (a few dozen kept tiles spread over the vocabulary) costs about one
// memory latency.  Mass and count of the upper side; its few tokens are also
// appended, in this warp's visiting order, to its own region of
// kSpecListCap / kWarps slots of `regions` (wrun counts them, also past the
// region's end).
constexpr int kRegion = kSpecListCap / kWarps;
constexpr int kFirstTiles = 3;
static_assert(kGemmBN == 2 * kStep, "a column tile is two 128-element steps");
__device__ __forceinline__ void first_pass(const float* et, const float* ftab, const int* kept,
                                           int nk, int V, float* regions, PassStats& ps,
                                           int& wrun) {
  const int l = lane_id();
  float* reg = regions + warp_id() * kRegion;
  wrun = 0;
  for (int j0 = warp_id(); j0 < nk; j0 += kFirstTiles * kWarps) {
    float4 v[kFirstTiles][2];
    float fm[kFirstTiles];
    int i0s[kFirstTiles];
#pragma unroll
    for (int u = 0; u < kFirstTiles; ++u) {
      const int j = j0 + u * kWarps;
      fm[u] = 0.f;
      i0s[u] = V;
      v[u][0] = v[u][1] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (j < nk) {  // warp-uniform
        const int t = kept[j];
        fm[u] = ftab[t];
        i0s[u] = t * kGemmBN + l * 4;
#pragma unroll
        for (int h = 0; h < 2; ++h)
          if (i0s[u] + h * kStep < V)
            v[u][h] = __ldg(reinterpret_cast<const float4*>(et + i0s[u] + h * kStep));
      }
    }
#pragma unroll
    for (int u = 0; u < kFirstTiles; ++u) {
      if (j0 + u * kWarps >= nk) break;  // warp-uniform
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int i0 = i0s[u] + h * kStep;
        const int nv = min(max(V - i0, 0), 4);
        const float e[4] = {v[u][h].x * fm[u], v[u][h].y * fm[u], v[u][h].z * fm[u],
                            v[u][h].w * fm[u]};
        bool ge[4];
        int k = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          ge[j] = j < nv && __float_as_uint(e[j]) >= kFirstMid;
          if (ge[j]) {
            ps.mass_ge += e[j];
            ++k;
          }
        }
        ps.cnt_ge += k;
        if (__any_sync(0xffffffffu, k > 0)) {
          const int incl = warp_incl_scan(k);
          int at = wrun + incl - k;
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (ge[j]) {
              if (at < kRegion) reg[at] = e[j];
              ++at;
            }
          wrun += __shfl_sync(0xffffffffu, incl, 31);
        }
      }
    }
  }
}

// Writes the row's tokens with key in [lo, lo + w) to dst in warp order,
// this warp from slot `run`, never past cnt.
__device__ __forceinline__ void row_compact(const float* et, const float* ftab, int V, uint32_t lo,
                                            uint32_t w, float* dst, int run, int cnt, int* status) {
  const int l = lane_id();
  constexpr int kStride = kWarps * kStep;
  for (int base = warp_id() * kStep; base < V; base += kUnroll * kStride) {
    float4 v[kUnroll];
    float fm[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int s0 = base + u * kStride, i0 = s0 + l * 4;
      fm[u] = s0 < V ? ftab[static_cast<unsigned>(s0) / kGemmBN] : 0.f;  // warp-uniform
      v[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (__float_as_uint(fm[u]) >= lo && i0 < V) v[u] = __ldg(reinterpret_cast<const float4*>(et + i0));
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      if (__float_as_uint(fm[u]) < lo) continue;  // warp-uniform: no candidate in this tile
      const int i0 = base + u * kStride + l * 4;
      float e[4] = {v[u].x * fm[u], v[u].y * fm[u], v[u].z * fm[u], v[u].w * fm[u]};
      bool keep[4];
      int k = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        keep[j] = i0 + j < V && __float_as_uint(e[j]) - lo < w;
        k += keep[j];
      }
      const int incl = warp_incl_scan(k);
      int at = run + incl - k;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (keep[j]) {
          MLS_CHECK(status, at < cnt);
          if (at < cnt) dst[at++] = e[j];
        }
      run += __shfl_sync(0xffffffffu, incl, 31);
    }
  }
}

// Block-wide combination; the per-warp counts stay in sh.n[w][1] (upper) and
// sh.n[w][2] (lower) for the compaction that may follow.
__device__ void reduce_pass(PassStats& s, Shared& sh) {
  const unsigned full = 0xffffffffu;
  s.mass_ge = warp_sum(s.mass_ge);
  s.cnt_ge = static_cast<int>(__reduce_add_sync(full, static_cast<unsigned>(s.cnt_ge)));
  s.cnt_lt = static_cast<int>(__reduce_add_sync(full, static_cast<unsigned>(s.cnt_lt)));
  s.min_ge = __reduce_min_sync(full, s.min_ge);
  s.max_ge = __reduce_max_sync(full, s.max_ge);
  s.min_lt = __reduce_min_sync(full, s.min_lt);
  s.max_lt = __reduce_max_sync(full, s.max_lt);
  __syncthreads();
  if (lane_id() == 0) {
    const int w = warp_id();
    sh.f[w][0] = s.mass_ge;
    sh.n[w][1] = s.cnt_ge;
    sh.n[w][2] = s.cnt_lt;
    sh.k[w][0] = s.min_ge;
    sh.k[w][1] = s.max_ge;
    sh.k[w][2] = s.min_lt;
    sh.k[w][3] = s.max_lt;
  }
  __syncthreads();
  if (warp_id() == 0) {
    const int l = lane_id();
    const bool has = l < kWarps;
    float m = has ? sh.f[l][0] : 0.f;
#pragma unroll
    for (int o = kWarps / 2; o > 0; o >>= 1) m += __shfl_xor_sync(full, m, o);
    const unsigned cg = __reduce_add_sync(full, has ? static_cast<unsigned>(sh.n[l][1]) : 0u);
    const unsigned cl = __reduce_add_sync(full, has ? static_cast<unsigned>(sh.n[l][2]) : 0u);
    const uint32_t a = __reduce_min_sync(full, has ? sh.k[l][0] : 0xffffffffu);
    const uint32_t b = __reduce_max_sync(full, has ? sh.k[l][1] : 0u);
    const uint32_t c = __reduce_min_sync(full, has ? sh.k[l][2] : 0xffffffffu);
    const uint32_t d = __reduce_max_sync(full, has ? sh.k[l][3] : 0u);
    if (l == 0) {
      sh.rf[0] = m;
      sh.rn[1] = static_cast<int>(cg);
      sh.rn[2] = static_cast<int>(cl);
      sh.rk[0] = a;
      sh.rk[1] = b;
      sh.rk[2] = c;
      sh.rk[3] = d;
    }
  }
  __syncthreads();
  s.mass_ge = sh.rf[0];
  s.cnt_ge = sh.rn[1];
  s.cnt_lt = sh.rn[2];
  s.min_ge = sh.rk[0];
  s.max_ge = sh.rk[1];
  s.min_lt = sh.rk[2];
  s.max_lt = sh.rk[3];
}

// After reduce_pass: each warp's first output slot when the survivors of
// side `side` (1 = upper, 2 = lower) are compacted in warp order.
__device__ __forceinline__ void warp_bases(int side, Shared& sh) {
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int w = 0; w < kWarps; ++w) {
      sh.wbase[w] = acc;
      acc += sh.n[w][side];
    }
  }
  __syncthreads();
}

struct RowNucleus {
  float m, S, b, kept;
  int c, eq;
};

// Exact boundary among the n <= kFinish candidates L (all keys in the current
// bracket; mass_hi is the mass above it): b = the largest candidate key whose
// mass(e >= key) = mass_hi + sum of the candidates >= it reaches the target
// (each candidate's sum is taken over L in index order, so it is monotone in
// the key), then the mass above b and the ties at b.
__device__ void finish_exact(const float* L, int n, float target, float mass_hi, uint32_t lo,
                             uint32_t& b, float& gt, int& eq, Shared& sh) {
  const int t = threadIdx.x;
  uint32_t kt = 0, best = 0;
  float et = 0.f;
  if (t < n) {
    et = L[t];
    kt = __float_as_uint(et);
    float M = 0.f;
    for (int j = 0; j < n; ++j) {
      const float ej = L[j];
      M += __float_as_uint(ej) >= kt ? ej : 0.f;
    }
    if (mass_hi + M >= target) best = kt + 1u;
  }
  best = block_max_u(best, sh);
  b = best ? best - 1u : lo;  // by rounding alone nothing may qualify: the bracket's bottom
  float part = (t < n && kt > b) ? et : 0.f;
  int ties = (t < n && kt == b) ? 1 : 0;
  block_sum2(part, ties, sh);
  gt = mass_hi + part;
  eq = ties;
}

// Nucleus of one row (e_t, per-tile stats st); writes f_t to fg.
__device__ RowNucleus nucleus(const float* et, const float* st, float* fg, long long V, int tiles,
                              float scale, float top_p, float* ftab, float* listA, float* listB,
                              Shared& sh, int* status) {
  RowNucleus r;
  row_stats(st, tiles, scale, ftab, fg, r.m, r.S, sh);
  const float target = top_p * r.S;
  // Invariant: mass(e >= lo) >= target > mass(e >= hi) = mass_hi; the
  // candidates are the elements with key in [lo, hi).
  uint32_t lo = 0u, hi = kOneKey + 1u;  // every e lies in [0, 1]
  float mass_hi = 0.f, gt = 0.f;
  int eq = 0;
  bool resolved = false;
  if (top_p < 1.f) {
    const float* list = nullptr;  // candidates in shared memory, once they fit
    int n_list = 0;
    bool done = false, probe2 = false;
    // ---- first pass: split at 2^-8
    {
      PassStats ps;
      int wrun = 0;
      // The kept-tile list lives in listB until the upper side is copied there.
      int* kept = reinterpret_cast<int*>(listB);
      const int nk = kept_tiles(ftab, tiles, kFirstMid, kept, sh);
      first_pass(et, ftab, kept, nk, static_cast<int>(V), listA, ps, wrun);
      if (lane_id() == 0) sh.wcnt[warp_id()] = wrun;
      reduce_pass(ps, sh);  // its barriers also publish wcnt
      int cnt;
      if (ps.mass_ge >= target) {
        cnt = ps.cnt_ge;
        lo = kFirstMid;
        // the upper side is in the warps' regions unless one overflowed
        bool fits = true;
        for (int w = 0; w < kWarps; ++w) fits = fits && sh.wcnt[w] <= kRegion;
        if (fits) {
          int at = 0;
          for (int w = 0; w < warp_id(); ++w) at += sh.wcnt[w];
          const float* reg = listA + warp_id() * kRegion;
          for (int i = lane_id(); i < sh.wcnt[warp_id()]; i += 32) listB[at + i] = reg[i];
          __syncthreads();
          list = listB;
          n_list = cnt;
        }
      } else {
        cnt = static_cast<int>(V) - ps.cnt_ge;
        mass_hi = ps.mass_ge;
        hi = kFirstMid;  // lo stays 0
        probe2 = true;
      }
      if (cnt == 0) {  // only by rounding, with top_p within an ulp of 1
        lo = 0u;
        done = true;
      } else if (list != nullptr && cnt <= kFinish) {
        finish_exact(list, n_list, target, mass_hi, lo, lo, gt, eq, sh);
        resolved = done = true;
      } else if (hi - lo <= 1u) {
        gt = mass_hi;
        eq = cnt;
        resolved = done = true;
      }
    }
    // ---- then bisection: untracked passes over the row, tracked ones over a list
    // Each pass at least halves hi - lo (< 2^30), so 32 passes always suffice.
    for (int pass = 1; !done && pass < 40; ++pass) {
      uint32_t mid = lo + (hi - lo) / 2u;
      if (probe2 && lo < kSecondMid && kSecondMid < hi) mid = kSecondMid;  // probe 2^-16 next
      probe2 = false;
      const bool track = list != nullptr;
      const uint32_t mo = mid - lo, wm = hi - mid;
      PassStats ps;
      if (list != nullptr) {
        for (int i = threadIdx.x; i < n_list; i += kThreads) ps.add<true>(list[i], lo, mo, wm);
      } else {
        row_pass<false>(et, ftab, static_cast<int>(V), lo, mo, wm, ps);
      }
      reduce_pass(ps, sh);
      int side, cnt;
      const uint32_t old_lo = lo;
      if (mass_hi + ps.mass_ge >= target) {
        side = 1;
        cnt = ps.cnt_ge;
        if (track) {
          lo = ps.min_ge;
          hi = ps.max_ge + 1u;
        } else {
          lo = mid;
        }
      } else {
        side = 2;
        cnt = ps.cnt_lt;
        mass_hi += ps.mass_ge;
        if (track) {
          lo = ps.min_lt;
          hi = ps.max_lt + 1u;
        } else {
          hi = mid;
        }
      }
      if (cnt == 0) {  // only by rounding, with top_p within an ulp of 1
        lo = old_lo;
        break;
      }
      if (hi - lo <= 1u) {  // one key left: the candidates are the ties at b
        gt = mass_hi;
        eq = cnt;
        resolved = true;
        break;
      }
      const bool finish = cnt <= kFinish;
      // Compact the survivors (keys in the new [lo, hi)) when that pays.
      if ((list == nullptr && cnt <= kSpecListCap) ||
          (list != nullptr && (2 * cnt <= n_list || (finish && cnt < n_list)))) {
        float* dst = list == listA ? listB : listA;
        warp_bases(side, sh);
        int run = sh.wbase[warp_id()];
        if (list == nullptr) {
          row_compact(et, ftab, static_cast<int>(V), lo, hi - lo, dst, run, cnt, status);
        } else {
          for (int base = warp_id() * 32; base < n_list; base += kThreads) {
            const int i = base + lane_id();
            float e = 0.f;
            bool keep = false;
            if (i < n_list) {
              e = list[i];
              keep = __float_as_uint(e) - lo < hi - lo;
            }
            const unsigned bal = __ballot_sync(0xffffffffu, keep);
            const int at = run + __popc(bal & ((1u << lane_id()) - 1u));
            if (keep) MLS_CHECK(status, at < cnt);
            if (keep && at < cnt) dst[at] = e;
            run += __popc(bal);
          }
        }
        __syncthreads();
        list = dst;
        n_list = cnt;
      }
      if (finish && list != nullptr && n_list == cnt) {
        finish_exact(list, n_list, target, mass_hi, lo, lo, gt, eq, sh);
        resolved = true;
        break;
      }
      MLS_CHECK(status, pass < 39);  // hi - lo at least halves each pass
    }
  }
  r.b = __uint_as_float(lo);
  if (!resolved) {  // top_p = 1, or the rounding exit: one more pass over the row
    float g = 0.f;
    int q = 0;
    for_row<kWarps>(et, ftab, V, [&](long long i0, const float4& v, long long n) {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (i0 + j < n) {
          const float e = comp(v, j);
          if (e > r.b) g += e;
          else if (e == r.b) ++q;
        }
    });
    block_sum2(g, q, sh);
    gt = g;
    eq = q;
  }
  r.eq = eq;
  int c = eq;
  if (top_p < 1.f && r.b > 0.f) {
    const float need = ceilf((target - gt) / r.b);
    c = need < 1.f ? 1 : (need >= static_cast<float>(eq) ? eq : static_cast<int>(need));
  }
  r.c = c;
  r.kept = gt + static_cast<float>(c) * r.b;
  return r;
}

// Nucleus probability of token x (block-wide: when x is tied at the boundary
// and only some ties are kept, its rank among them is counted).
template <int NW>
__device__ float prob_of(const float* et, const float* ftab, long long V, const RowNucleus& n,
                         int x, SharedT<NW>& sh) {
  const float e = et[x] * ftab[x / kGemmBN];
  bool member = e > n.b;
  if (e == n.b) {
    if (n.c >= n.eq) {
      member = true;
    } else {
      float unused = 0.f;
      int below = 0;
      for_row<NW>(et, ftab, V, [&](long long i0, const float4& v, long long cnt) {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (i0 + j < x && i0 + j < cnt && comp(v, j) == n.b) ++below;
      });
      block_sum2(unused, below, sh);
      member = below < n.c;
    }
  }
  return member ? e * (1.f / n.kept) : 0.f;
}

__device__ __forceinline__ void store_state(float* st, const RowNucleus& n) {
  st[0] = n.m;
  st[1] = n.b;
  st[2] = n.kept;
  st[3] = __int_as_float(n.c);
  st[4] = __int_as_float(n.eq);
  st[5] = n.S;
}

__device__ __forceinline__ RowNucleus load_state(const float* st) {
  RowNucleus n;
  n.m = st[0];
  n.b = st[1];
  n.kept = st[2];
  n.c = __float_as_int(st[3]);
  n.eq = __float_as_int(st[4]);
  n.S = st[5];
  return n;
}

// Shared memory of spec_row_kernel: the row's f_t table, then two lists.
__host__ __device__ __forceinline__ size_t row_smem(int tiles) {
  return sizeof(float) * ((static_cast<size_t>(tiles) + 3) / 4 * 4 + 2 * kSpecListCap);
}

// One CTA per logits row: rows [0, B (gamma + 1)) are the verifier's, the
// rest the draft's.  Leaves the row's nucleus state and its f_t table.
__global__ void __launch_bounds__(kThreads, 4) spec_row_kernel(const SpecParams p) {
  extern __shared__ __align__(16) float smem[];
  __shared__ Shared sh;
  const int tiles_pad = (p.tiles + 3) / 4 * 4;
  float* ftab = smem;
  float* listA = smem + tiles_pad;
  float* listB = listA + kSpecListCap;
  const long long Pv = static_cast<long long>(p.B) * (p.gamma + 1);
  const long long sld = 2LL * p.tiles;
  long long r = blockIdx.x;
  const bool verifier = r < Pv;
  if (!verifier) r -= Pv;
  const float* et = (verifier ? p.ev : p.ed) + r * p.ldz;
  const RowNucleus n = nucleus(et, (verifier ? p.stats_v : p.stats_d) + r * sld,
                               (verifier ? p.f_v : p.f_d) + r * p.tiles, p.V, p.tiles, p.scale,
                               p.top_p, ftab, listA, listB, sh, p.status);
  if (threadIdx.x == 0) store_state((verifier ? p.state_v : p.state_d) + r * kSpecStateWords, n);
}

// ------------------------------------------------------------------ sampling
// Inverse-CDF sampling in index order over steps of 128 tokens: one pass gives
// every step's mass (warps take steps w, w + 16, ...), one thread accumulates
// them in index order, and one warp walks the step in which the cumulative
// passes u * total.

// Unnormalised probabilities e of the lane's 4 tokens from i0 (zeros past V).
__device__ __forceinline__ float4 load_e(const float* et, const float* ftab, long long i0,
                                         long long V) {
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
  if (i0 < V) {
    v = __ldg(reinterpret_cast<const float4*>(et + i0));
    const float fm = ftab[i0 / kGemmBN];
    v.x *= fm;
    v.y *= fm;
    v.z *= fm;
    v.w *= fm;
  }
  return v;
}

// Nucleus probabilities of those 4 tokens; rank0 (warp-uniform) counts the
// ties at b before this step in index order (only read when some ties are out).
__device__ __forceinline__ void probs4(const float4& v, long long i0, long long V,
                                       const RowNucleus& n, float inv, int rank0, float (&pr)[4]) {
  float e[4];
  bool valid[4];
  int ties = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    valid[j] = i0 + j < V;
    e[j] = comp(v, j);
    ties += valid[j] && e[j] == n.b;
  }
  if (n.c >= n.eq) {
#pragma unroll
    for (int j = 0; j < 4; ++j) pr[j] = (valid[j] && e[j] >= n.b) ? e[j] * inv : 0.f;
    return;
  }
  const int incl = warp_incl_scan(ties);
  int rank = rank0 + incl - ties;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    bool in = valid[j] && e[j] > n.b;
    if (valid[j] && e[j] == n.b) in = rank++ < n.c;
    pr[j] = in ? e[j] * inv : 0.f;
  }
}

// In-place inclusive prefix sum of a[0, n) in index order: each thread sums a
// contiguous run of entries, the runs' totals are scanned across the block
// (warps by shuffles, then warp 0 over the warp totals), and each run is
// rewritten from its offset.  Fixed order, so deterministic.
template <int NW>
__device__ void block_inclusive_scan(float* a, int n, SharedT<NW>& sh) {
  const int per = (n + (NW * 32) - 1) / (NW * 32);
  const int b0 = min(n, static_cast<int>(threadIdx.x) * per), b1 = min(n, b0 + per);
  float t = 0.f;
  for (int i = b0; i < b1; ++i) t += a[i];
  const float incl = warp_incl_scan(t);
  __syncthreads();
  if (lane_id() == 31) sh.f[warp_id()][1] = incl;
  __syncthreads();
  if (warp_id() == 0) {
    const float wt = lane_id() < NW ? sh.f[lane_id()][1] : 0.f;
    const float wi = warp_incl_scan(wt);
    if (lane_id() < NW) sh.f[lane_id()][0] = wi - wt;  // exclusive warp offsets
  }
  __syncthreads();
  float run = sh.f[warp_id()][0] + (incl - t);
  for (int i = b0; i < b1; ++i) {
    run += a[i];
    a[i] = run;
  }
  __syncthreads();
}

// Per step: the ties at b, then (thread 0, in index order) their exclusive prefix.
template <int NW>
__device__ void step_tie_bases(const float* et, const float* ftab, const RowNucleus& n, long long V,
                               int nsteps, int* base) {
  const int w = warp_id(), l = lane_id();
  for (int st = w; st < nsteps; st += NW) {
    const long long i0 = static_cast<long long>(st) * kStep + l * 4;
    if (ftab[static_cast<long long>(st) * kStep / kGemmBN] < n.b) {  // no e reaches b here
      if (l == 0) base[st] = 0;
      continue;
    }
    const float4 v = load_e(et, ftab, i0, V);
    int t = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) t += i0 + j < V && comp(v, j) == n.b;
    t = static_cast<int>(__reduce_add_sync(0xffffffffu, static_cast<unsigned>(t)));
    if (l == 0) base[st] = t;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int run = 0;
    for (int st = 0; st < nsteps; ++st) {
      const int t = base[st];
      base[st] = run;
      run += t;
    }
  }
  __syncthreads();
}

// sample(r, u) over r_v = max(0, p_v - q_v) (have_q) or r_v = p_v; -1 when r
// is all zero.  cum: nsteps floats; tp/tq: nsteps ints each; live: one int
// per column tile.
template <int NW>
__device__ int sample(const float* ep, const float* fp, const RowNucleus& np, const float* eq,
                      const float* fq, const RowNucleus& nq, bool have_q, long long V, float u,
                      float* cum, int* tp, int* tq, int* live, SharedT<NW>& sh, int* status) {
  const int nsteps = static_cast<int>((V + kStep - 1) / kStep);
  const int w = warp_id(), l = lane_id();
  const float ip = 1.f / np.kept, iq = have_q ? 1.f / nq.kept : 0.f;
  const bool part_p = np.c < np.eq, part_q = have_q && nq.c < nq.eq;
  if (part_p) step_tie_bases<NW>(ep, fp, np, V, nsteps, tp);
  if (part_q) step_tie_bases<NW>(eq, fq, nq, V, nsteps, tq);
  // Mass of every step.  p is 0 where e < b, so only the tiles whose maximum
  // f_t reaches b (listed in tile order) are read; warp w takes live tiles w,
  // w + NW, ..., one tile (two steps, p and q) per round with all four loads
  // in flight.  The other steps' masses are 0.
  for (int st = threadIdx.x; st < nsteps; st += NW * 32) cum[st] = 0.f;
  const int nlive = kept_tiles(fp, (nsteps * kStep + kGemmBN - 1) / kGemmBN,
                               __float_as_uint(np.b), live, sh);  // its barriers publish cum
  for (int j = w; j < nlive; j += NW) {
    const int t = live[j];
    float4 vp[2], vq[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const long long i0 = static_cast<long long>(t) * kGemmBN + h * kStep + l * 4;
      vp[h] = load_e(ep, fp, i0, V);
      vq[h] = have_q ? load_e(eq, fq, i0, V) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int st = t * (kGemmBN / kStep) + h;
      if (st >= nsteps) break;  // warp-uniform
      const long long i0 = static_cast<long long>(st) * kStep + l * 4;
      float a[4], c[4] = {0.f, 0.f, 0.f, 0.f};
      probs4(vp[h], i0, V, np, ip, part_p ? tp[st] : 0, a);
      if (have_q) probs4(vq[h], i0, V, nq, iq, part_q ? tq[st] : 0, c);
      float m = 0.f;
#pragma unroll
      for (int j2 = 0; j2 < 4; ++j2) m += fmaxf(0.f, a[j2] - c[j2]);
      m = warp_sum(m);
      if (l == 0) cum[st] = m;
    }
  }
  __syncthreads();
  block_inclusive_scan(cum, nsteps, sh);
  const float total = cum[nsteps - 1];
  if (!(total > 0.f)) return -1;
  const float want = u * total;
  if (w == 0) {
    // the first step whose cumulative passes want (and that has mass)
    int owner = -1;
    for (int s0 = 0; s0 < nsteps && owner < 0; s0 += 32) {
      const int st = s0 + l;
      const float prev = st > 0 && st < nsteps ? cum[st - 1] : 0.f;
      const bool hit = st < nsteps && cum[st] > want && cum[st] > prev;
      const unsigned bal = __ballot_sync(0xffffffffu, hit);
      if (bal) owner = s0 + __ffs(bal) - 1;
    }
    float before = 0.f;
    if (owner < 0) {  // rounding put want at the total: the last step with mass
      for (int st = nsteps - 1; st >= 0 && owner < 0; --st)
        if (cum[st] > (st > 0 ? cum[st - 1] : 0.f)) owner = st;
      before = -INFINITY;  // pick its last token with mass
      MLS_CHECK(status, owner >= 0);
      if (owner < 0) owner = 0;
    } else {
      before = owner > 0 ? cum[owner - 1] : 0.f;
    }
    const long long i0 = static_cast<long long>(owner) * kStep + l * 4;
    float a[4], c[4] = {0.f, 0.f, 0.f, 0.f};
    probs4(load_e(ep, fp, i0, V), i0, V, np, ip, part_p ? tp[owner] : 0, a);
    if (have_q) probs4(load_e(eq, fq, i0, V), i0, V, nq, iq, part_q ? tq[owner] : 0, c);
    float r[4], lane_sum = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      r[j] = fmaxf(0.f, a[j] - c[j]);
      lane_sum += r[j];
    }
    const float incl = warp_incl_scan(lane_sum);
    float run = before + (incl - lane_sum);
    long long my_found = -1, my_last = -1;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (r[j] > 0.f) {
        my_last = i0 + j;
        run += r[j];
        if (my_found < 0 && run > want) my_found = i0 + j;
      }
    const unsigned fb = __ballot_sync(0xffffffffu, my_found >= 0);
    const unsigned lb = __ballot_sync(0xffffffffu, my_last >= 0);
    long long res = static_cast<long long>(owner) * kStep;  // unreachable fallbacks
    if (fb) res = __shfl_sync(0xffffffffu, my_found, __ffs(fb) - 1);
    else if (lb) res = __shfl_sync(0xffffffffu, my_last, 31 - __clz(lb));
    if (l == 0) sh.n[0][0] = static_cast<int>(res);
  }
  __syncthreads();
  return sh.n[0][0];
}

// Greedy: the verifier's argmax of row `pos` from its tile (max, argmax) pairs.
template <int NW>
__device__ int row_argmax(const float* st, int tiles, SharedT<NW>& sh) {
  float mv = -INFINITY;
  int mi = 0;
  for (int t = threadIdx.x; t < tiles; t += (NW * 32))
    if (st[2 * t] > mv) {
      mv = st[2 * t];
      mi = __float_as_int(st[2 * t + 1]);
    }
  block_argmax(mv, mi, sh);
  return mi;
}

__global__ void __launch_bounds__(kSampleWarps * 32) spec_sample_kernel(const SpecParams p) {
  extern __shared__ __align__(16) float smem[];
  __shared__ SharedT<kSampleWarps> sh;
  const int b = blockIdx.x, G1 = p.gamma + 1;
  const long long sld = 2LL * p.tiles;
  int k = 0, next = -1;
  if (p.greedy) {
    for (;; ++k) {
      const int best = row_argmax(p.stats_v + (static_cast<long long>(b) * G1 + k) * sld, p.tiles, sh);
      if (k == p.gamma || p.draft[static_cast<long long>(b) * p.gamma + k] != best) {
        next = best;
        break;
      }
    }
  } else {
    const int nsteps = static_cast<int>((p.V + kStep - 1) / kStep);
    float* fp = smem;
    float* fq = fp + p.tiles;
    float* cum = fq + p.tiles;
    int* tp = reinterpret_cast<int*>(cum + nsteps);
    int* tq = tp + nsteps;
    int* live = tq + nsteps;  // the sampler's live tiles
    int* acc = live + p.tiles;  // per drafted position: 1 accepted, 0 rejected, 2 undecided
    // Acceptance of every drafted token, in parallel: q(x) and p(x) from the
    // rows' nucleus states; a token tied at a boundary of which only some
    // ties are kept needs its rank among them (a pass over the row, below).
    for (int i = threadIdx.x; i < p.gamma; i += kSampleWarps * 32) {
      const long long pos_d = static_cast<long long>(b) * p.gamma + i, pos_v = static_cast<long long>(b) * G1 + i;
      const int x = p.draft[pos_d];
      int f = 0;
      if (x >= 0 && x < p.V) {
        const RowNucleus nq = load_state(p.state_d + pos_d * kSpecStateWords);
        const RowNucleus np = load_state(p.state_v + pos_v * kSpecStateWords);
        const float eq = p.ed[pos_d * p.ldz + x] * p.f_d[pos_d * p.tiles + x / kGemmBN];
        const float ep = p.ev[pos_v * p.ldz + x] * p.f_v[pos_v * p.tiles + x / kGemmBN];
        const bool rank_q = eq == nq.b && nq.c < nq.eq, rank_p = ep == np.b && np.c < np.eq;
        if (rank_q || rank_p) {
          f = 2;
        } else {
          const float qx = eq >= nq.b ? eq * (1.f / nq.kept) : 0.f;
          const float px = ep >= np.b ? ep * (1.f / np.kept) : 0.f;
          f = qx > 0.f && p.u[pos_v * 2] * qx < px;
        }
      }
      acc[i] = f;
    }
    __syncthreads();
    for (; k < p.gamma; ++k) {
      int f = acc[k];
      if (f == 2) {  // block-wide: rank of x among the ties at the boundary
        const long long pos_d = static_cast<long long>(b) * p.gamma + k, pos_v = static_cast<long long>(b) * G1 + k;
        const int x = p.draft[pos_d];
        for (int t = threadIdx.x; t < p.tiles; t += kSampleWarps * 32) {
          fq[t] = p.f_d[pos_d * p.tiles + t];
          fp[t] = p.f_v[pos_v * p.tiles + t];
        }
        __syncthreads();
        const float qx = prob_of(p.ed + pos_d * p.ldz, fq, p.V,
                                 load_state(p.state_d + pos_d * kSpecStateWords), x, sh);
        const float px = prob_of(p.ev + pos_v * p.ldz, fp, p.V,
                                 load_state(p.state_v + pos_v * kSpecStateWords), x, sh);
        f = qx > 0.f && p.u[pos_v * 2] * qx < px;
        __syncthreads();
      }
      if (!f) break;
    }
    const long long pos_v = static_cast<long long>(b) * G1 + k;
    const RowNucleus np = load_state(p.state_v + pos_v * kSpecStateWords);
    const float* ev = p.ev + pos_v * p.ldz;
    for (int t = threadIdx.x; t < p.tiles; t += kSampleWarps * 32) fp[t] = p.f_v[pos_v * p.tiles + t];
    const float u = p.u[pos_v * 2 + 1];
    if (k < p.gamma) {
      const long long pos_d = static_cast<long long>(b) * p.gamma + k;
      const RowNucleus nq = load_state(p.state_d + pos_d * kSpecStateWords);
      for (int t = threadIdx.x; t < p.tiles; t += kSampleWarps * 32) fq[t] = p.f_d[pos_d * p.tiles + t];
      __syncthreads();
      next = sample(ev, fp, np, p.ed + pos_d * p.ldz, fq, nq, true, p.V, u, cum, tp, tq, live, sh,
                    p.status);
    }
    __syncthreads();
    if (next < 0) next = sample(ev, fp, np, ev, fp, np, false, p.V, u, cum, tp, tq, live, sh, p.status);
    if (next < 0) next = static_cast<int>(p.V - 1);  // unreachable: the maximum has e = 1
  }
  if (threadIdx.x == 0) {
    p.n_accepted[b] = k;
    p.next_token[b] = next;
  }
}

size_t sample_smem(long long V, int tiles, int gamma) {
  const long long nsteps = (V + kStep - 1) / kStep;
  return sizeof(float) * (3 * static_cast<size_t>(tiles) + 3 * static_cast<size_t>(nsteps) +
                          static_cast<size_t>(gamma));
}

}  // namespace

cudaError_t setup_spec_kernels() {
  cudaError_t e = cudaFuncSetAttribute(spec_row_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(row_smem(kSpecMaxTiles)));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(
      spec_sample_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
      static_cast<int>(sample_smem(static_cast<long long>(kSpecMaxTiles) * kGemmBN, kSpecMaxTiles,
                                   kSpecMaxGamma)));
}

cudaError_t launch_spec_rows(const SpecParams& p, cudaStream_t s) {
  const long long rows = static_cast<long long>(p.B) * (2 * p.gamma + 1);
  if (rows <= 0 || p.greedy) return cudaSuccess;
  spec_row_kernel<<<static_cast<unsigned>(rows), kThreads, row_smem(p.tiles), s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_spec_sample(const SpecParams& p, cudaStream_t s) {
  if (p.B <= 0) return cudaSuccess;
  spec_sample_kernel<<<p.B, kSampleWarps * 32, p.greedy ? 0 : sample_smem(p.V, p.tiles, p.gamma), s>>>(p);
  return cudaGetLastError();
}

}  // namespace mls
