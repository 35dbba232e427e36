// Row reductions of the forward pass, the token count of the backward and an
// fp32 transpose (used only for fp32 inputs, whose tf32 GEMMs read K-major copies).
//
// merge_kernel: a block of 8 warps combines, for 8 to 64 tokens, the partial row
// states that the head kernel wrote per (CTA, half tile) into
//   lse_m    = logsumexp(z_m)            CE_m = lse_m - z_m[y]
//   lset_m   = logsumexp(z_m / tau)
//   E_q[z_m] = sum_v q_v z_m[v]          from A_m / S_t (q = softmax(z_t / tau))
//   Ld_m     = lset_m - E_q[z_m] / tau   (Eq. 2: -sum_v q_v log softmax(z_m/tau)_v)
//   H(q)     = lset_t - E_q[z_t] / tau,  KL_m = Ld_m - H(q); the teacher's
//              sum is kept relative to its maximum so H(q) has no cancellation
//   L_m      = (1 - alpha) CE_m + alpha Ld_m  (Eq. 3),  L_t = CE_t
// and the block's share of sum_t sum_m w_m L_m[t].  Partials are merged by
// rescaling each one from its own running maximum to the row maximum.
// final_kernel adds the block shares in a fixed order (deterministic) and
// divides by N, the number of tokens whose target lies in [0, V).
#include <climits>

#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

__device__ __forceinline__ double block_sum_double(double v, double* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) sh[w] = v;
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0)
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s += sh[i];
  return s;  // valid in thread 0
}

// A block of 8 warps merges 8 * (8 / kWT) consecutive tokens: each group of 8
// tokens (an octet) takes kWT warps, i.e. 4 * kWT partial slots per token.
// Lane l of warp w takes token (l mod 8) of octet w / kWT and the partials
// k = 4 (w mod kWT) + l / 8, k + 4 kWT, ...: the 8 lanes of a group read 32
// consecutive bytes (one sector) of each (partial, field, sub-model).  kWT
// follows the number of partials (merge_warps_per_octet), so few partials
// do not leave most lanes idle.  Pass 1 takes every sub-model's row maximum,
// pass 2 its sums.  The partials of a token are combined in a fixed order
// (within a lane, across the 4 lane groups by butterflies, across the octet's
// warps in warp order), and the block's share of the loss over its octets in
// octet order, so results are deterministic.
constexpr int kMergeWarps = 8;

template <int kWT>
__global__ void __launch_bounds__(kMergeWarps * 32, 4) merge_kernel(const __grid_constant__ MergeParams p) {
  constexpr int kOct = kMergeWarps / kWT;  // token octets per block
  constexpr int kSlots = 4 * kWT;          // partial slots per token
  __shared__ float sh_f[4][kMergeWarps][kMaxModels][8];  // max, then s1, st, acc, zy
  __shared__ int sh_am[kMergeWarps][kMaxModels][8];
  __shared__ double sh_c[kOct][2];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = lane & 7, grp = lane >> 3;  // token within the octet, partial group
  const int oct = w / kWT, ww = w % kWT;    // octet, warp within the octet
  const long long T = p.T;
  const long long t = (static_cast<long long>(blockIdx.x) * kOct + oct) * 8 + j;
  const bool live = t < T;
  const long long MT = static_cast<long long>(p.M) * T;
  const long long PS = kPartFields * MT;  // stride between partials
  const int tc = p.teacher;
  const int k0 = 4 * ww + grp;

  // ---- pass 1: row maxima of every sub-model
  float mx[kMaxModels];
#pragma unroll
  for (int m = 0; m < kMaxModels; ++m) mx[m] = -INFINITY;
  if (live)
    for (int k = k0; k < p.nparts; k += kSlots) {
#pragma unroll
      for (int m = 0; m < kMaxModels; ++m)
        if (m < p.M) mx[m] = fmaxf(mx[m], p.part[k * PS + kPartMax * MT + m * T + t]);
    }
#pragma unroll
  for (int m = 0; m < kMaxModels; ++m) {
    mx[m] = fmaxf(mx[m], __shfl_xor_sync(0xffffffffu, mx[m], 8));
    mx[m] = fmaxf(mx[m], __shfl_xor_sync(0xffffffffu, mx[m], 16));
    if (grp == 0) sh_f[0][w][m][j] = mx[m];
  }
  __syncthreads();
#pragma unroll
  for (int m = 0; m < kMaxModels; ++m) {
    float v = -INFINITY;
    for (int q = 0; q < kWT; ++q) v = fmaxf(v, sh_f[0][oct * kWT + q][m][j]);
    mx[m] = v;
  }
  float mT = -INFINITY;
#pragma unroll
  for (int m = 0; m < kMaxModels; ++m)
    if (m == tc) mT = mx[m];
  __syncthreads();  // sh_f[0] is reused below

  // ---- pass 2: sums.  The teacher's weighted sum is relative to its own
  // maximum: B_k = sum q~ (z - m_k) log2(e)/tau; moving it to the row maximum
  // mT adds (m_k - mT) log2(e)/tau per unit of weight before the weights are
  // rescaled.  A student's A_k is relative to the teacher's maximum of the
  // same partial.
  float s1[kMaxModels], st[kMaxModels], acc[kMaxModels], zy[kMaxModels];
  int am[kMaxModels];
#pragma unroll
  for (int m = 0; m < kMaxModels; ++m) {
    s1[m] = st[m] = acc[m] = zy[m] = 0.f;
    am[m] = INT_MAX;
  }
  if (live)
    for (int k = k0; k < p.nparts; k += kSlots) {
      const float mtk = p.part[k * PS + kPartMax * MT + static_cast<long long>(tc) * T + t];
#pragma unroll
      for (int m = 0; m < kMaxModels; ++m) {
        if (m >= p.M) continue;
        const float* P = p.part + k * PS + static_cast<long long>(m) * T + t;
        const float mk = P[kPartMax * MT];
        if (m == tc) {
          if (mk != -INFINITY) {
            const float f1 = exp2f((mk - mT) * p.L1);
            const float ft = exp2f((mk - mT) * p.Ltau);
            const float stk = P[kPartSumTau * MT];
            s1[m] += P[kPartSum1 * MT] * f1;
            st[m] += stk * ft;
            acc[m] += (P[kPartAcc * MT] + (mk - mT) * p.Ltau * stk) * ft;
          }
        } else {
          if (mk != -INFINITY) {
            s1[m] += P[kPartSum1 * MT] * exp2f((mk - mx[m]) * p.L1);
            st[m] += P[kPartSumTau * MT] * exp2f((mk - mx[m]) * p.Ltau);
          }
          if (mtk != -INFINITY) acc[m] += P[kPartAcc * MT] * exp2f((mtk - mT) * p.Ltau);
        }
        zy[m] += P[kPartTarget * MT];
        if (mk == mx[m]) am[m] = min(am[m], __float_as_int(P[kPartArgmax * MT]));
      }
    }
#pragma unroll
  for (int m = 0; m < kMaxModels; ++m) {
#pragma unroll
    for (int o = 8; o <= 16; o <<= 1) {
      s1[m] += __shfl_xor_sync(0xffffffffu, s1[m], o);
      st[m] += __shfl_xor_sync(0xffffffffu, st[m], o);
      acc[m] += __shfl_xor_sync(0xffffffffu, acc[m], o);
      zy[m] += __shfl_xor_sync(0xffffffffu, zy[m], o);
      am[m] = min(am[m], __shfl_xor_sync(0xffffffffu, am[m], o));
    }
    if (grp == 0) {
      sh_f[0][w][m][j] = s1[m];
      sh_f[1][w][m][j] = st[m];
      sh_f[2][w][m][j] = acc[m];
      sh_f[3][w][m][j] = zy[m];
      sh_am[w][m][j] = am[m];
    }
  }
  __syncthreads();

  // ---- the octet's first warp, lanes 0-7: one token each
  double contrib = 0.0, cnt = 0.0;
  if (ww == 0 && lane < 8 && live) {
#pragma unroll
    for (int m = 0; m < kMaxModels; ++m) {
      float a = 0.f, b = 0.f, c = 0.f, d = 0.f;
      int e = INT_MAX;
      for (int q = 0; q < kWT; ++q) {
        const int wq = oct * kWT + q;
        a += sh_f[0][wq][m][j];
        b += sh_f[1][wq][m][j];
        c += sh_f[2][wq][m][j];
        d += sh_f[3][wq][m][j];
        e = min(e, sh_am[wq][m][j]);
      }
      s1[m] = a;
      st[m] = b;
      acc[m] = c;
      zy[m] = d;
      am[m] = e;
    }
    const int y = p.y[t];
    const bool bad = y >= p.V;
    if (bad) atomicOr(p.status, kStatusBadTarget);
    const bool valid = y >= 0 && !bad;
    const float invtau = 1.0f / p.tau;
    float s1T = 0.f, stT = 0.f, bT = 0.f, zT = 0.f;
    int amT = INT_MAX;
#pragma unroll
    for (int m = 0; m < kMaxModels; ++m)
      if (m == tc) {
        s1T = s1[m];
        stT = st[m];
        bT = acc[m];
        zT = zy[m];
        amT = am[m];
      }
    const float lseT = mT + logf(s1T);
    const float lsetT = mT * invtau + logf(stT);
    // H(q) = log S - E_q[(z - mT)/tau]; both terms are >= 0
    const float HqT = logf(stT) - bT / (stT * p.L1);
#pragma unroll
    for (int m = 0; m < kMaxModels; ++m) {
      if (m >= p.M) continue;
      float lse, lset, ce, ld, kl, L;
      int amm;
      if (m == tc) {
        lse = lseT;
        lset = lsetT;
        ce = lseT - zT;
        ld = HqT;
        kl = 0.f;
        L = ce;
        amm = amT;
      } else {
        lse = mx[m] + logf(s1[m]);
        lset = mx[m] * invtau + logf(st[m]);
        ce = lse - zy[m];
        ld = lset - (acc[m] / stT) * invtau;
        kl = ld - HqT;
        L = (1.f - p.alpha) * ce + p.alpha * ld;
        amm = am[m];
      }
      if (!valid) ce = ld = kl = L = 0.f;
      const long long o = static_cast<long long>(m) * T + t;
      p.tok_loss[o] = L;
      if (p.tok_diag) {
        p.tok_diag[o] = ce;
        p.tok_diag[MT + o] = ld;
        p.tok_diag[2 * MT + o] = kl;
      }
      if (p.argmax) p.argmax[o] = amm;
      p.stats[o] = lse;
      p.stats[MT + o] = lset;
      contrib += static_cast<double>(p.w[m]) * static_cast<double>(L);
    }
    cnt = valid ? 1.0 : 0.0;
  }
  // the block's share, over its tokens in a fixed order: within each octet,
  // then over the octets
#pragma unroll
  for (int o = 4; o > 0; o >>= 1) {
    contrib += __shfl_down_sync(0xffffffffu, contrib, o);
    cnt += __shfl_down_sync(0xffffffffu, cnt, o);
  }
  if (ww == 0 && lane == 0) {
    sh_c[oct][0] = contrib;
    sh_c[oct][1] = cnt;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double bs = 0.0, bc = 0.0;
    for (int o = 0; o < kOct; ++o) {
      bs += sh_c[o][0];
      bc += sh_c[o][1];
    }
    p.block_sum[blockIdx.x] = bs;
    p.block_cnt[blockIdx.x] = static_cast<long long>(bc);
  }
}

constexpr int kFinalThreads = 256;

__global__ void __launch_bounds__(kFinalThreads)
    final_kernel(const double* __restrict__ bsum, const long long* __restrict__ bcnt, int n,
                 float* loss) {
  __shared__ double sh[kFinalThreads / 32];
  double s = 0.0, c = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    s += bsum[i];
    c += static_cast<double>(bcnt[i]);
  }
  const double S = block_sum_double(s, sh);
  const double C = block_sum_double(c, sh);
  if (threadIdx.x == 0) *loss = C > 0.0 ? static_cast<float>(S / C) : 0.f;
}

constexpr int kCountThreads = 1024;

__global__ void __launch_bounds__(kCountThreads)
    count_kernel(const int* __restrict__ y, long long T, long long V, float* inv_n, int* status) {
  __shared__ double sh[kCountThreads / 32];
  double c = 0.0;
  bool bad = false;
  for (long long i = threadIdx.x; i < T; i += blockDim.x) {
    const int v = y[i];
    if (v >= V) bad = true;
    else if (v >= 0) c += 1.0;
  }
  if (bad) atomicOr(status, kStatusBadTarget);
  const double C = block_sum_double(c, sh);
  if (threadIdx.x == 0) *inv_n = C > 0.0 ? static_cast<float>(1.0 / C) : 0.f;
}

// out[c][r] = in[r][c] for an fp32 [rows, cols] matrix, through 32x32 tiles.
constexpr int kTile = 32;
__global__ void __launch_bounds__(kTile * 8)
    transpose_kernel(const float* __restrict__ in, long long rows, long long cols, long long ld_in,
                     float* __restrict__ out, long long ld_out) {
  __shared__ float tile[kTile][kTile + 1];
  const long long r0 = static_cast<long long>(blockIdx.y) * kTile;
  const long long c0 = static_cast<long long>(blockIdx.x) * kTile;
  for (int i = threadIdx.y; i < kTile; i += blockDim.y) {
    const long long r = r0 + i, c = c0 + threadIdx.x;
    tile[i][threadIdx.x] = (r < rows && c < cols) ? in[r * ld_in + c] : 0.f;
  }
  __syncthreads();
  for (int i = threadIdx.y; i < kTile; i += blockDim.y) {
    const long long c = c0 + i, r = r0 + threadIdx.x;
    if (c < cols && r < rows) out[c * ld_out + r] = tile[threadIdx.x][i];
  }
}

}  // namespace

cudaError_t launch_transpose(const float* in, long long rows, long long cols, long long ld_in,
                             float* out, long long ld_out, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return cudaSuccess;
  const dim3 grid(static_cast<unsigned>((cols + kTile - 1) / kTile),
                  static_cast<unsigned>((rows + kTile - 1) / kTile));
  transpose_kernel<<<grid, dim3(kTile, 8), 0, s>>>(in, rows, cols, ld_in, out, ld_out);
  return cudaGetLastError();
}

cudaError_t launch_merge(const MergeParams& p, int blocks, cudaStream_t s) {
  if (blocks <= 0) return cudaSuccess;
  switch (merge_warps_per_octet(p.nparts)) {
    case 1: merge_kernel<1><<<blocks, kMergeWarps * 32, 0, s>>>(p); break;
    case 2: merge_kernel<2><<<blocks, kMergeWarps * 32, 0, s>>>(p); break;
    default: merge_kernel<8><<<blocks, kMergeWarps * 32, 0, s>>>(p); break;
  }
  return cudaGetLastError();
}

cudaError_t launch_final(const double* block_sum, const long long* block_cnt, int nblocks,
                         float* loss, cudaStream_t s) {
  final_kernel<<<1, kFinalThreads, 0, s>>>(block_sum, block_cnt, nblocks, loss);
  return cudaGetLastError();
}

cudaError_t launch_count(const int* y, long long T, long long V, float* inv_n, int* status,
                         cudaStream_t s) {
  count_kernel<<<1, kCountThreads, 0, s>>>(y, T, V, inv_n, status);
  return cudaGetLastError();
}

}  // namespace mls
