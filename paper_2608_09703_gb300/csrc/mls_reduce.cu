// Row reductions of the forward pass, the token count of the backward and an
// fp32 transpose (used only for fp32 inputs, whose tf32 GEMMs read K-major copies).
//
// merge_kernel: one warp per token combines the partial row states that the
// head kernel wrote per (CTA, half tile) into
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

__device__ __forceinline__ float warp_max_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One warp per token: lane k takes partials k, k + 32, ...; warp reductions
// (butterflies, so every lane holds the same result and the order is fixed)
// combine them, and lane 0 writes the token's outputs.
__global__ void __launch_bounds__(kMergeTokens * 32) merge_kernel(const __grid_constant__ MergeParams p) {
  __shared__ double sh_sum[kMergeTokens], sh_cnt[kMergeTokens];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long t = static_cast<long long>(blockIdx.x) * kMergeTokens + w;
  double contrib = 0.0, cnt = 0.0;
  if (t < p.T) {  // warp-uniform
    const long long T = p.T;
    const long long MT = static_cast<long long>(p.M) * T;
    const long long PS = kPartFields * MT;  // stride between partials
    const int y = p.y[t];
    const bool bad = y >= p.V;
    if (bad && lane == 0) atomicOr(p.status, kStatusBadTarget);
    const bool valid = y >= 0 && !bad;
    const float invtau = 1.0f / p.tau;
    const int tc = p.teacher;
    const float* Pt = p.part + static_cast<long long>(tc) * T + t;

    // teacher: row maximum, sums at tau = 1 and tau, teacher-weighted sum B
    float mT = -INFINITY;
    for (int k = lane; k < p.nparts; k += 32) mT = fmaxf(mT, Pt[k * PS + kPartMax * MT]);
    mT = warp_max_f(mT);
    // The teacher's weighted sum is relative to its own maximum:
    // B_k = sum q~ (z - m_k) log2(e)/tau; moving it to the row maximum mT adds
    // (m_k - mT) log2(e)/tau per unit of weight before the weights are rescaled.
    float s1T = 0.f, stT = 0.f, bT = 0.f, zT = 0.f;
    int amT = INT_MAX;
    for (int k = lane; k < p.nparts; k += 32) {
      const float* P = Pt + k * PS;
      const float mk = P[kPartMax * MT];
      if (mk != -INFINITY) {
        const float f1 = exp2f((mk - mT) * p.L1);
        const float ft = exp2f((mk - mT) * p.Ltau);
        const float stk = P[kPartSumTau * MT];
        s1T += P[kPartSum1 * MT] * f1;
        stT += stk * ft;
        bT += (P[kPartAcc * MT] + (mk - mT) * p.Ltau * stk) * ft;
      }
      zT += P[kPartTarget * MT];
      if (mk == mT) amT = min(amT, __float_as_int(P[kPartArgmax * MT]));
    }
    s1T = warp_sum_f(s1T);
    stT = warp_sum_f(stT);
    bT = warp_sum_f(bT);
    zT = warp_sum_f(zT);
    amT = __reduce_min_sync(0xffffffffu, amT);
    const float lseT = mT + logf(s1T);
    const float lsetT = mT * invtau + logf(stT);
    // H(q) = log S - E_q[(z - mT)/tau]; both terms are >= 0
    const float HqT = logf(stT) - bT / (stT * p.L1);

    for (int m = 0; m < p.M; ++m) {
      float lse, lset, ce, ld, kl, L;
      int am;
      if (m == tc) {
        lse = lseT;
        lset = lsetT;
        ce = lseT - zT;
        ld = HqT;
        kl = 0.f;
        L = ce;
        am = amT;
      } else {
        const float* Pm = p.part + static_cast<long long>(m) * T + t;
        float mm = -INFINITY;
        for (int k = lane; k < p.nparts; k += 32) mm = fmaxf(mm, Pm[k * PS + kPartMax * MT]);
        mm = warp_max_f(mm);
        float s1 = 0.f, st = 0.f, A = 0.f, zy = 0.f;
        am = INT_MAX;
        for (int k = lane; k < p.nparts; k += 32) {
          const float* P = Pm + k * PS;
          const float mk = P[kPartMax * MT];
          if (mk != -INFINITY) {
            s1 += P[kPartSum1 * MT] * exp2f((mk - mm) * p.L1);
            st += P[kPartSumTau * MT] * exp2f((mk - mm) * p.Ltau);
          }
          const float mtk = Pt[k * PS + kPartMax * MT];  // the teacher max this A is relative to
          if (mtk != -INFINITY) A += P[kPartAcc * MT] * exp2f((mtk - mT) * p.Ltau);
          zy += P[kPartTarget * MT];
          if (mk == mm) am = min(am, __float_as_int(P[kPartArgmax * MT]));
        }
        s1 = warp_sum_f(s1);
        st = warp_sum_f(st);
        A = warp_sum_f(A);
        zy = warp_sum_f(zy);
        am = __reduce_min_sync(0xffffffffu, am);
        lse = mm + logf(s1);
        lset = mm * invtau + logf(st);
        ce = lse - zy;
        ld = lset - (A / stT) * invtau;
        kl = ld - HqT;
        L = (1.f - p.alpha) * ce + p.alpha * ld;
      }
      if (!valid) ce = ld = kl = L = 0.f;
      if (lane == 0) {
        const long long o = static_cast<long long>(m) * T + t;
        p.tok_loss[o] = L;
        if (p.tok_diag) {
          p.tok_diag[o] = ce;
          p.tok_diag[MT + o] = ld;
          p.tok_diag[2 * MT + o] = kl;
        }
        if (p.argmax) p.argmax[o] = am;
        p.stats[o] = lse;
        p.stats[MT + o] = lset;
      }
      contrib += static_cast<double>(p.w[m]) * static_cast<double>(L);
    }
    cnt = valid ? 1.0 : 0.0;
  }
  if (lane == 0) {
    sh_sum[w] = contrib;
    sh_cnt[w] = cnt;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double bs = 0.0, bc = 0.0;
    for (int i = 0; i < kMergeTokens; ++i) {
      bs += sh_sum[i];
      bc += sh_cnt[i];
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
  merge_kernel<<<blocks, kMergeTokens * 32, 0, s>>>(p);
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
