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
//   spec_position_kernel (one CTA per position, sampling only) finds each
//     row's nucleus: the boundary value b = the largest e with
//     mass(e' >= b) >= top_p S, by bisection over the bit patterns of e
//     (non-negative floats order like their bits), each pass narrowing the
//     bracket to its surviving keys; survivors are compacted into shared memory
//     once they fit and the last <= 256 are resolved exactly; then the c
//     lowest-index tokens with e == b that the cumulative needs.  It then
//     decides acceptance of the drafted token of that position.
//   spec_sample_kernel (one CTA per sequence) takes the first rejection and
//     samples by inverse CDF in index order, each warp walking a contiguous
//     segment of the vocabulary; for greedy it reduces the tile argmaxes.
// Every reduction has a fixed order, so a call is deterministic.
#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kStep = 128;              // elements one warp covers per float4 step
constexpr int kUnroll = 4;              // independent float4 loads in flight per lane
constexpr int kFinish = 256;            // candidates resolved exactly
constexpr uint32_t kInfKey = 0x7f800000u;
constexpr uint32_t kFirstMid = 0x3b800000u;  // 2^-8: first split of the bracket [0, inf)
constexpr size_t kPositionSmem = sizeof(float) * (kSpecMaxTiles + 2 * kSpecListCap);
static_assert(kFinish <= kThreads, "one candidate per thread in the exact finish");

struct Shared {
  float f[kWarps][2];
  int n[kWarps][3];
  uint32_t k[kWarps][4];
  int wbase[kWarps];
};

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

// Block-wide (max value, lowest index attaining it).
__device__ void block_argmax(float& v, int& idx, Shared& sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, idx, o);
    if (ov > v || (ov == v && oi < idx)) {
      v = ov;
      idx = oi;
    }
  }
  __syncthreads();
  if (lane_id() == 0) {
    sh.f[warp_id()][0] = v;
    sh.n[warp_id()][0] = idx;
  }
  __syncthreads();
  v = sh.f[0][0];
  idx = sh.n[0][0];
  for (int w = 1; w < kWarps; ++w)
    if (sh.f[w][0] > v || (sh.f[w][0] == v && sh.n[w][0] < idx)) {
      v = sh.f[w][0];
      idx = sh.n[w][0];
    }
}

// Block sums of a float and an int (fixed order: lanes by a butterfly, warps 0..15).
__device__ void block_sum2(float& f, int& n, Shared& sh) {
  f = warp_sum(f);
  n = static_cast<int>(__reduce_add_sync(0xffffffffu, static_cast<unsigned>(n)));
  __syncthreads();
  if (lane_id() == 0) {
    sh.f[warp_id()][0] = f;
    sh.n[warp_id()][0] = n;
  }
  __syncthreads();
  f = 0.f;
  n = 0;
  for (int w = 0; w < kWarps; ++w) {
    f += sh.f[w][0];
    n += sh.n[w][0];
  }
}

__device__ uint32_t block_max_u(uint32_t v, Shared& sh) {
  v = __reduce_max_sync(0xffffffffu, v);
  __syncthreads();
  if (lane_id() == 0) sh.k[warp_id()][0] = v;
  __syncthreads();
  uint32_t r = 0;
  for (int w = 0; w < kWarps; ++w) r = max(r, sh.k[w][0]);
  return r;
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
template <typename F>
__device__ __forceinline__ void for_row(const float* et, const float* ftab, long long V, F&& f) {
  const int l = lane_id();
  constexpr long long kStride = static_cast<long long>(kWarps) * kStep;
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
// split at mid: mass and count of the upper side, count of the lower side,
// and the smallest and largest key on each side.
struct PassStats {
  float mass_ge = 0.f;
  int cnt_ge = 0, cnt_lt = 0;
  uint32_t min_ge = 0xffffffffu, max_ge = 0u, min_lt = 0xffffffffu, max_lt = 0u;
  __device__ __forceinline__ void add(float e, uint32_t lo, uint32_t mid, uint32_t hi) {
    const uint32_t key = __float_as_uint(e);
    if (key < lo || key >= hi) return;
    if (key >= mid) {
      mass_ge += e;
      ++cnt_ge;
      min_ge = min(min_ge, key);
      max_ge = max(max_ge, key);
    } else {
      ++cnt_lt;
      min_lt = min(min_lt, key);
      max_lt = max(max_lt, key);
    }
  }
};

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
  PassStats r;
  for (int w = 0; w < kWarps; ++w) {
    r.mass_ge += sh.f[w][0];
    r.cnt_ge += sh.n[w][1];
    r.cnt_lt += sh.n[w][2];
    r.min_ge = min(r.min_ge, sh.k[w][0]);
    r.max_ge = max(r.max_ge, sh.k[w][1]);
    r.min_lt = min(r.min_lt, sh.k[w][2]);
    r.max_lt = max(r.max_lt, sh.k[w][3]);
  }
  s = r;
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
                              Shared& sh) {
  RowNucleus r;
  row_stats(st, tiles, scale, ftab, fg, r.m, r.S, sh);
  const float target = top_p * r.S;
  // Invariant: mass(e >= lo) >= target > mass(e >= hi) = mass_hi; the
  // candidates are the elements with key in [lo, hi).
  uint32_t lo = 0u, hi = kInfKey;
  float mass_hi = 0.f, gt = 0.f;
  int eq = 0;
  bool resolved = false;
  if (top_p < 1.f) {
    const float* list = nullptr;  // candidates in shared memory, once they fit
    int n_list = 0;
    // Each pass at least halves hi - lo (< 2^31), so 33 passes always suffice.
    for (int pass = 0; pass < 40; ++pass) {
      const uint32_t mid = pass == 0 ? kFirstMid : lo + (hi - lo) / 2u;
      PassStats ps;
      if (list == nullptr) {
        for_row(et, ftab, V, [&](long long i0, const float4& v, long long n) {
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (i0 + j < n) ps.add(comp(v, j), lo, mid, hi);
        });
      } else {
        for (int i = threadIdx.x; i < n_list; i += kThreads) ps.add(list[i], lo, mid, hi);
      }
      reduce_pass(ps, sh);
      int side, cnt;
      const uint32_t old_lo = lo;
      if (mass_hi + ps.mass_ge >= target) {
        side = 1;
        cnt = ps.cnt_ge;
        lo = ps.min_ge;
        hi = ps.max_ge + 1u;
      } else {
        side = 2;
        cnt = ps.cnt_lt;
        mass_hi += ps.mass_ge;
        lo = ps.min_lt;
        hi = ps.max_lt + 1u;
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
          for_row(et, ftab, V, [&](long long i0, const float4& v, long long n) {
            int k = 0;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint32_t key = __float_as_uint(comp(v, j));
              k += i0 + j < n && key >= lo && key < hi;
            }
            const int incl = warp_incl_scan(k);
            int at = run + incl - k;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint32_t key = __float_as_uint(comp(v, j));
              if (i0 + j < n && key >= lo && key < hi && at < cnt) dst[at++] = comp(v, j);
            }
            run += __shfl_sync(0xffffffffu, incl, 31);
          });
        } else {
          for (int base = warp_id() * 32; base < n_list; base += kThreads) {
            const int i = base + lane_id();
            float e = 0.f;
            bool keep = false;
            if (i < n_list) {
              e = list[i];
              const uint32_t key = __float_as_uint(e);
              keep = key >= lo && key < hi;
            }
            const unsigned bal = __ballot_sync(0xffffffffu, keep);
            const int at = run + __popc(bal & ((1u << lane_id()) - 1u));
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
    }
  }
  r.b = __uint_as_float(lo);
  if (!resolved) {  // top_p = 1, or the rounding exit: one more pass over the row
    float g = 0.f;
    int q = 0;
    for_row(et, ftab, V, [&](long long i0, const float4& v, long long n) {
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
__device__ float prob_of(const float* et, const float* ftab, long long V, const RowNucleus& n,
                         int x, Shared& sh) {
  const float e = et[x] * ftab[x / kGemmBN];
  bool member = e > n.b;
  if (e == n.b) {
    if (n.c >= n.eq) {
      member = true;
    } else {
      float unused = 0.f;
      int below = 0;
      for_row(et, ftab, V, [&](long long i0, const float4& v, long long cnt) {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (i0 + j < x && i0 + j < cnt && comp(v, j) == n.b) ++below;
      });
      block_sum2(unused, below, sh);
      member = below < n.c;
    }
  }
  return member ? e / n.kept : 0.f;
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

__global__ void __launch_bounds__(kThreads, 2) spec_position_kernel(const SpecParams p) {
  extern __shared__ __align__(16) float smem[];
  __shared__ Shared sh;
  float* ftab = smem;
  float* listA = smem + kSpecMaxTiles;
  float* listB = listA + kSpecListCap;
  const int G1 = p.gamma + 1;
  const int b = blockIdx.x / G1, i = blockIdx.x % G1;
  const long long pos_v = static_cast<long long>(b) * G1 + i;
  const long long sld = 2LL * p.tiles;
  const float* ev = p.ev + pos_v * p.ldz;
  const RowNucleus np = nucleus(ev, p.stats_v + pos_v * sld, p.f_v + pos_v * p.tiles, p.V,
                                p.tiles, p.scale, p.top_p, ftab, listA, listB, sh);
  if (threadIdx.x == 0) store_state(p.state_v + pos_v * kSpecStateWords, np);
  if (i == p.gamma) return;
  const int x = p.draft[static_cast<long long>(b) * p.gamma + i];
  float px = 0.f;
  if (x >= 0 && x < p.V) px = prob_of(ev, ftab, p.V, np, x, sh);
  __syncthreads();  // ftab is rewritten for the draft row
  const long long pos_d = static_cast<long long>(b) * p.gamma + i;
  const float* ed = p.ed + pos_d * p.ldz;
  const RowNucleus nq = nucleus(ed, p.stats_d + pos_d * sld, p.f_d + pos_d * p.tiles, p.V,
                                p.tiles, p.scale, p.top_p, ftab, listA, listB, sh);
  if (threadIdx.x == 0) store_state(p.state_d + pos_d * kSpecStateWords, nq);
  int ok = 0;
  if (x >= 0 && x < p.V) {
    const float qx = prob_of(ed, ftab, p.V, nq, x, sh);
    ok = qx > 0.f && p.u[pos_v * 2] * qx < px;
  }
  if (threadIdx.x == 0) p.acc[pos_v] = ok;
}

// ------------------------------------------------------------------ sampling
// Per-warp contiguous segments of the vocabulary, in index order.
struct Segment {
  long long begin, end;
};
__device__ __forceinline__ Segment my_segment(long long V) {
  const long long steps = (V + kStep - 1) / kStep;
  const long long per = (steps + kWarps - 1) / kWarps * kStep;
  const long long b = min(V, per * warp_id());
  return {b, min(V, b + per)};
}

// Nucleus probabilities of the lane's 4 elements from i0 in one step of a
// segment ending at `end`; `tie_run` (warp-uniform) counts the ties at b
// before this step in index order.
__device__ __forceinline__ void probs4(const float* et, const float* ftab, const RowNucleus& n,
                                       long long i0, long long end, int& tie_run, float (&pr)[4]) {
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
  if (i0 < end) {
    v = __ldg(reinterpret_cast<const float4*>(et + i0));
    const float fm = ftab[i0 / kGemmBN];
    v.x *= fm;
    v.y *= fm;
    v.z *= fm;
    v.w *= fm;
  }
  const float inv = 1.f / n.kept;
  float e[4];
  bool valid[4];
  int ties = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    valid[j] = i0 + j < end;
    e[j] = comp(v, j);
    ties += valid[j] && e[j] == n.b;
  }
  if (n.c >= n.eq) {
#pragma unroll
    for (int j = 0; j < 4; ++j) pr[j] = (valid[j] && e[j] >= n.b) ? e[j] * inv : 0.f;
    return;
  }
  const int incl = warp_incl_scan(ties);
  int rank = tie_run + incl - ties;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    bool in = valid[j] && e[j] > n.b;
    if (valid[j] && e[j] == n.b) in = rank++ < n.c;
    pr[j] = in ? e[j] * inv : 0.f;
  }
  tie_run += __shfl_sync(0xffffffffu, incl, 31);
}

// Ties at b in this warp's segment (the bases of the tie ranks).
__device__ int segment_ties(const float* et, const float* ftab, const RowNucleus& n,
                            const Segment& sg) {
  int t = 0;
  for (long long base = sg.begin; base < sg.end; base += kStep) {
    const long long i0 = base + lane_id() * 4;
    if (i0 < sg.end) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(et + i0));
      const float fm = ftab[i0 / kGemmBN];
#pragma unroll
      for (int j = 0; j < 4; ++j) t += (i0 + j < sg.end) && comp(v, j) * fm == n.b;
    }
  }
  return static_cast<int>(__reduce_add_sync(0xffffffffu, static_cast<unsigned>(t)));
}

// sample(r, u) over r_v = max(0, p_v - q_v) (have_q) or r_v = p_v; -1 when r
// is all zero.
__device__ int sample(const float* ep, const float* fp, const RowNucleus& np, const float* eq,
                      const float* fq, const RowNucleus& nq, bool have_q, long long V, float u,
                      Shared& sh) {
  const Segment sg = my_segment(V);
  const int w = warp_id(), l = lane_id();
  int base_p = 0, base_q = 0;
  const bool tp = np.c < np.eq, tq = have_q && nq.c < nq.eq;
  if (tp || tq) {
    const int cp = tp ? segment_ties(ep, fp, np, sg) : 0;
    const int cq = tq ? segment_ties(eq, fq, nq, sg) : 0;
    __syncthreads();
    if (l == 0) {
      sh.n[w][1] = cp;
      sh.n[w][2] = cq;
    }
    __syncthreads();
    for (int k = 0; k < w; ++k) {
      base_p += sh.n[k][1];
      base_q += sh.n[k][2];
    }
  }
  // mass of each warp's segment
  float mine = 0.f;
  {
    int rp = base_p, rq = base_q;
    for (long long base = sg.begin; base < sg.end; base += kStep) {
      float a[4], c[4] = {0.f, 0.f, 0.f, 0.f};
      probs4(ep, fp, np, base + l * 4, sg.end, rp, a);
      if (have_q) probs4(eq, fq, nq, base + l * 4, sg.end, rq, c);
#pragma unroll
      for (int j = 0; j < 4; ++j) mine += fmaxf(0.f, a[j] - c[j]);
    }
  }
  mine = warp_sum(mine);
  __syncthreads();
  if (l == 0) sh.f[w][0] = mine;
  __syncthreads();
  float total = 0.f;
  for (int k = 0; k < kWarps; ++k) total += sh.f[k][0];
  if (!(total > 0.f)) return -1;
  const float want = u * total;
  // the segment in which the cumulative passes want, and the mass before it
  int owner = -1;
  float before = 0.f;
  {
    float incl = 0.f;
    for (int k = 0; k < kWarps; ++k) {
      const float next = incl + sh.f[k][0];
      if (owner < 0 && next > want && sh.f[k][0] > 0.f) {
        owner = k;
        before = incl;
      }
      incl = next;
    }
    if (owner < 0) {  // rounding put want past the end: the last token with mass
      for (int k = kWarps - 1; k >= 0 && owner < 0; --k)
        if (sh.f[k][0] > 0.f) owner = k;
      before = -INFINITY;
    }
  }
  __syncthreads();
  if (w == owner) {
    int rp = base_p, rq = base_q;
    float cum = before;
    long long found = -1, last = -1;
    for (long long base = sg.begin; base < sg.end && found < 0; base += kStep) {
      float a[4], c[4] = {0.f, 0.f, 0.f, 0.f};
      const long long i0 = base + l * 4;
      probs4(ep, fp, np, i0, sg.end, rp, a);
      if (have_q) probs4(eq, fq, nq, i0, sg.end, rq, c);
      float r[4], lane_sum = 0.f;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        r[j] = fmaxf(0.f, a[j] - c[j]);
        lane_sum += r[j];
      }
      const float incl = warp_incl_scan(lane_sum);
      float run = cum + (incl - lane_sum);
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
      if (fb) found = __shfl_sync(0xffffffffu, my_found, __ffs(fb) - 1);
      if (lb) last = __shfl_sync(0xffffffffu, my_last, 31 - __clz(lb));
      cum += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (l == 0) sh.n[0][0] = static_cast<int>(found >= 0 ? found : last);
  }
  __syncthreads();
  return sh.n[0][0];
}

// Greedy: the verifier's argmax of row `pos` from its tile (max, argmax) pairs.
__device__ int row_argmax(const float* st, int tiles, Shared& sh) {
  float mv = -INFINITY;
  int mi = 0;
  for (int t = threadIdx.x; t < tiles; t += kThreads)
    if (st[2 * t] > mv) {
      mv = st[2 * t];
      mi = __float_as_int(st[2 * t + 1]);
    }
  block_argmax(mv, mi, sh);
  return mi;
}

__global__ void __launch_bounds__(kThreads) spec_sample_kernel(const SpecParams p) {
  __shared__ Shared sh;
  __shared__ float fp[kSpecMaxTiles], fq[kSpecMaxTiles];
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
    while (k < p.gamma && p.acc[static_cast<long long>(b) * G1 + k]) ++k;
    const long long pos_v = static_cast<long long>(b) * G1 + k;
    const RowNucleus np = load_state(p.state_v + pos_v * kSpecStateWords);
    const float* ev = p.ev + pos_v * p.ldz;
    for (int t = threadIdx.x; t < p.tiles; t += kThreads) fp[t] = p.f_v[pos_v * p.tiles + t];
    const float u = p.u[pos_v * 2 + 1];
    if (k < p.gamma) {
      const long long pos_d = static_cast<long long>(b) * p.gamma + k;
      const RowNucleus nq = load_state(p.state_d + pos_d * kSpecStateWords);
      for (int t = threadIdx.x; t < p.tiles; t += kThreads) fq[t] = p.f_d[pos_d * p.tiles + t];
      __syncthreads();
      next = sample(ev, fp, np, p.ed + pos_d * p.ldz, fq, nq, true, p.V, u, sh);
    }
    __syncthreads();
    if (next < 0) next = sample(ev, fp, np, ev, fp, np, false, p.V, u, sh);
    if (next < 0) next = static_cast<int>(p.V - 1);  // unreachable: the maximum has e = 1
  }
  if (threadIdx.x == 0) {
    p.n_accepted[b] = k;
    p.next_token[b] = next;
  }
}

}  // namespace

cudaError_t setup_spec_kernels() {
  return cudaFuncSetAttribute(spec_position_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(kPositionSmem));
}

cudaError_t launch_spec_position(const SpecParams& p, cudaStream_t s) {
  const long long blocks = static_cast<long long>(p.B) * (p.gamma + 1);
  if (blocks <= 0 || p.greedy) return cudaSuccess;
  spec_position_kernel<<<static_cast<unsigned>(blocks), kThreads, kPositionSmem, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_spec_sample(const SpecParams& p, cudaStream_t s) {
  if (p.B <= 0) return cudaSuccess;
  spec_sample_kernel<<<p.B, kThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace mls
