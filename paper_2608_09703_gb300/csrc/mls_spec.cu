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
// The logits of the few verify positions are produced by the tensor-core GEMM
// (fp32, one row per position).  Here, in units e_v = 2^((z_v - max) log2(e) / T):
//   spec_position_kernel (one CTA per position) finds each row's nucleus: the
//     boundary value b = the largest e with mass(e' >= b) >= top_p * S, by
//     bisection over the bit patterns of e (non-negative floats order like
//     their bits), each pass narrowing the bracket to its surviving keys and
//     compacting the survivors into shared memory once they fit; then the c
//     lowest-index tokens with e == b that the cumulative needs.  It then
//     decides acceptance of the drafted token of that position.
//   spec_sample_kernel (one CTA per sequence) takes the first rejection and
//     samples by inverse CDF in index order, each warp walking a contiguous
//     segment of the vocabulary.
// Every reduction has a fixed order, so a call is deterministic.
#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kStep = 128;  // elements one warp covers per float4 step
constexpr uint32_t kInfKey = 0x7f800000u;

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

__device__ __forceinline__ float e_of(float z, float m, float scale) {
  return fast_exp2((z - m) * scale);
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

// Visits a logits row of V elements, warp w taking the 128-element steps
// w, w + 16, ...: `f(i0, z4, V)` gets the lane's 4 consecutive elements from
// index i0 (entries at or past V are not meaningful).  The loop is
// warp-uniform, so f may use warp collectives.  Rows are 16-byte aligned and
// padded to a multiple of 4 elements.
template <typename F>
__device__ __forceinline__ void for_row(const float* z, long long V, F&& f) {
  const int l = lane_id();
  for (long long base = static_cast<long long>(warp_id()) * kStep; base < V;
       base += static_cast<long long>(kWarps) * kStep) {
    const long long i0 = base + l * 4;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i0 < V) v = __ldg(reinterpret_cast<const float4*>(z + i0));
    f(i0, v, V);
  }
}

// Statistics of one bisection pass over the candidates with key in [lo, hi),
// split at mid: mass and count of the upper side, count of the lower side,
// and the smallest and largest key on each side.
struct PassStats {
  float mass_ge = 0.f;
  int cnt_ge = 0, cnt_lt = 0;
  uint32_t min_ge = 0xffffffffu, max_ge = 0u, min_lt = 0xffffffffu, max_lt = 0u;
  __device__ __forceinline__ void add(float e, uint32_t key, uint32_t lo, uint32_t mid, uint32_t hi) {
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

// Nucleus of softmax(z / T) for one logits row (scale = log2(e) / T); listA
// and listB hold `cap` floats each.
__device__ RowNucleus nucleus(const float* z, long long V, float scale, float top_p, float* listA,
                              float* listB, int cap, Shared& sh) {
  RowNucleus r;
  {
    float mv = -INFINITY;
    int mi = 0;
    for_row(z, V, [&](long long i0, const float4& v, long long n) {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (i0 + j < n && comp(v, j) > mv) {
          mv = comp(v, j);
          mi = static_cast<int>(i0 + j);
        }
    });
    block_argmax(mv, mi, sh);
    r.m = mv;
  }
  {
    float s = 0.f;
    int unused = 0;
    for_row(z, V, [&](long long i0, const float4& v, long long n) {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (i0 + j < n) s += e_of(comp(v, j), r.m, scale);
    });
    block_sum2(s, unused, sh);
    r.S = s;
  }
  const float target = top_p * r.S;
  // Invariant: mass(e >= lo) >= target > mass(e >= hi) = mass_hi; the
  // candidates are the elements with key in [lo, hi).
  uint32_t lo = 0u, hi = kInfKey;
  float mass_hi = 0.f;
  if (top_p < 1.f) {
    const float* list = nullptr;  // candidates in shared memory, once they fit
    int n_list = 0;
    // Each pass at least halves hi - lo (< 2^31), so 32 passes always suffice.
    for (int pass = 0; pass < 40 && hi - lo > 1u; ++pass) {
      const uint32_t mid = lo + (hi - lo) / 2u;
      PassStats ps;
      if (list == nullptr) {
        for_row(z, V, [&](long long i0, const float4& v, long long n) {
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (i0 + j < n) {
              const float e = e_of(comp(v, j), r.m, scale);
              ps.add(e, __float_as_uint(e), lo, mid, hi);
            }
        });
      } else {
        for (int i = threadIdx.x; i < n_list; i += kThreads) {
          const float e = list[i];
          ps.add(e, __float_as_uint(e), lo, mid, hi);
        }
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
      if (hi - lo <= 1u) break;
      // Compact the survivors (keys in the new [lo, hi)) when that pays.
      const bool from_row = list == nullptr && cnt <= cap;
      const bool shrink = list != nullptr && 2 * cnt <= n_list;
      if (from_row || shrink) {
        float* dst = list == listA ? listB : listA;
        warp_bases(side, sh);
        int run = sh.wbase[warp_id()];
        if (from_row) {
          for_row(z, V, [&](long long i0, const float4& v, long long n) {
            float e[4];
            int k = 0;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              e[j] = e_of(comp(v, j), r.m, scale);
              const uint32_t key = __float_as_uint(e[j]);
              const bool keep = i0 + j < n && key >= lo && key < hi;
              k += keep;
              if (!keep) e[j] = -1.f;
            }
            const int incl = warp_incl_scan(k);
            int at = run + incl - k;
#pragma unroll
            for (int j = 0; j < 4; ++j)
              if (e[j] >= 0.f && at < cnt) dst[at++] = e[j];
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
    }
  }
  r.b = __uint_as_float(lo);
  // Mass strictly above b, and the tokens tied at b.
  float gt = 0.f;
  int eq = 0;
  for_row(z, V, [&](long long i0, const float4& v, long long n) {
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (i0 + j < n) {
        const float e = e_of(comp(v, j), r.m, scale);
        if (e > r.b) gt += e;
        else if (e == r.b) ++eq;
      }
  });
  block_sum2(gt, eq, sh);
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
__device__ float prob_of(const float* z, long long V, float scale, const RowNucleus& n, int x,
                         Shared& sh) {
  const float e = e_of(z[x], n.m, scale);
  bool member = e > n.b;
  if (e == n.b) {
    if (n.c >= n.eq) {
      member = true;
    } else {
      float unused = 0.f;
      int below = 0;
      for_row(z, V, [&](long long i0, const float4& v, long long cnt) {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (i0 + j < x && i0 + j < cnt && e_of(comp(v, j), n.m, scale) == n.b) ++below;
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
  extern __shared__ __align__(16) float lists[];
  __shared__ Shared sh;
  const int G1 = p.gamma + 1;
  const int b = blockIdx.x / G1, i = blockIdx.x % G1;
  const long long pos_v = static_cast<long long>(b) * G1 + i;
  const float* zv = p.zv + pos_v * p.ldz;
  if (p.greedy) {
    float mv = -INFINITY;
    int mi = 0;
    for_row(zv, p.V, [&](long long i0, const float4& v, long long n) {
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (i0 + j < n && comp(v, j) > mv) {
          mv = comp(v, j);
          mi = static_cast<int>(i0 + j);
        }
    });
    block_argmax(mv, mi, sh);
    if (threadIdx.x == 0) {
      p.tok[pos_v] = mi;
      p.acc[pos_v] = i < p.gamma && p.draft[static_cast<long long>(b) * p.gamma + i] == mi;
    }
    return;
  }
  const RowNucleus np = nucleus(zv, p.V, p.scale, p.top_p, lists, lists + p.cap, p.cap, sh);
  if (threadIdx.x == 0) store_state(p.state_v + pos_v * kSpecStateWords, np);
  if (i == p.gamma) return;
  const long long pos_d = static_cast<long long>(b) * p.gamma + i;
  const float* zd = p.zd + pos_d * p.ldz;
  const RowNucleus nq = nucleus(zd, p.V, p.scale, p.top_p, lists, lists + p.cap, p.cap, sh);
  if (threadIdx.x == 0) store_state(p.state_d + pos_d * kSpecStateWords, nq);
  const int x = p.draft[pos_d];
  int ok = 0;
  if (x >= 0 && x < p.V) {
    const float qx = prob_of(zd, p.V, p.scale, nq, x, sh);
    const float px = prob_of(zv, p.V, p.scale, np, x, sh);
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
__device__ __forceinline__ void probs4(const float* z, const RowNucleus& n, float scale,
                                       long long i0, long long end, int& tie_run, float (&pr)[4]) {
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
  if (i0 < end) v = __ldg(reinterpret_cast<const float4*>(z + i0));
  const float inv = 1.f / n.kept;
  float e[4];
  bool valid[4];
  int ties = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    valid[j] = i0 + j < end;
    e[j] = e_of(comp(v, j), n.m, scale);
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
__device__ int segment_ties(const float* z, const RowNucleus& n, float scale, const Segment& sg) {
  int t = 0;
  for (long long base = sg.begin; base < sg.end; base += kStep) {
    const long long i0 = base + lane_id() * 4;
    if (i0 < sg.end) {
      const float4 v = __ldg(reinterpret_cast<const float4*>(z + i0));
#pragma unroll
      for (int j = 0; j < 4; ++j) t += (i0 + j < sg.end) && e_of(comp(v, j), n.m, scale) == n.b;
    }
  }
  return static_cast<int>(__reduce_add_sync(0xffffffffu, static_cast<unsigned>(t)));
}

// sample(r, u) over r_v = max(0, p_v - q_v) (have_q) or r_v = p_v; -1 when r
// is all zero.
__device__ int sample(const float* zp, const RowNucleus& np, const float* zq, const RowNucleus& nq,
                      bool have_q, float scale, long long V, float u, Shared& sh) {
  const Segment sg = my_segment(V);
  const int w = warp_id(), l = lane_id();
  int base_p = 0, base_q = 0;
  const bool tp = np.c < np.eq, tq = have_q && nq.c < nq.eq;
  if (tp || tq) {
    const int cp = tp ? segment_ties(zp, np, scale, sg) : 0;
    const int cq = tq ? segment_ties(zq, nq, scale, sg) : 0;
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
      probs4(zp, np, scale, base + l * 4, sg.end, rp, a);
      if (have_q) probs4(zq, nq, scale, base + l * 4, sg.end, rq, c);
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
      probs4(zp, np, scale, i0, sg.end, rp, a);
      if (have_q) probs4(zq, nq, scale, i0, sg.end, rq, c);
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

__global__ void __launch_bounds__(kThreads) spec_sample_kernel(const SpecParams p) {
  __shared__ Shared sh;
  const int b = blockIdx.x, G1 = p.gamma + 1;
  int k = 0;
  while (k < p.gamma && p.acc[static_cast<long long>(b) * G1 + k]) ++k;
  const long long pos_v = static_cast<long long>(b) * G1 + k;
  int next;
  if (p.greedy) {
    next = p.tok[pos_v];
  } else {
    const RowNucleus np = load_state(p.state_v + pos_v * kSpecStateWords);
    const float* zv = p.zv + pos_v * p.ldz;
    const float u = p.u[pos_v * 2 + 1];
    next = -1;
    if (k < p.gamma) {
      const long long pos_d = static_cast<long long>(b) * p.gamma + k;
      const RowNucleus nq = load_state(p.state_d + pos_d * kSpecStateWords);
      next = sample(zv, np, p.zd + pos_d * p.ldz, nq, true, p.scale, p.V, u, sh);
    }
    if (next < 0) next = sample(zv, np, zv, np, false, p.scale, p.V, u, sh);
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
                              static_cast<int>(2 * kSpecListCap * sizeof(float)));
}

cudaError_t launch_spec_position(const SpecParams& p, cudaStream_t s) {
  const long long blocks = static_cast<long long>(p.B) * (p.gamma + 1);
  if (blocks <= 0) return cudaSuccess;
  const size_t smem = p.greedy ? 0 : 2 * static_cast<size_t>(p.cap) * sizeof(float);
  spec_position_kernel<<<static_cast<unsigned>(blocks), kThreads, smem, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_spec_sample(const SpecParams& p, cudaStream_t s) {
  if (p.B <= 0) return cudaSuccess;
  spec_sample_kernel<<<p.B, kThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace mls
