// Forward-only evaluation metrics between the sub-models of a suite
// (paper Sec. 3.2.2: pairwise KL divergence and top-1 agreement; App. A plots
// KL(p_student || p_teacher)).  For every token and ordered pair (s, j):
//   KL(p_s || p_j) = E_{p_s}[z_s - z_j] - (lse_s - lse_j)
// with p = softmax(z) at temperature 1.  The logits are never stored.
//
// A CTA pair owns 256 tokens and a strided set of 128-column vocabulary tiles.
// For each tile the even CTA issues pair MMAs (cta_group::2, 256x128xK) for
// every sub-model into its own 128 TMEM columns, so all M <= 4 logit tiles are
// resident together; the epilogue then reads them chunk by chunk and
// accumulates, per sub-model s, the running max, sum_v exp(z_s - max_s) and
// D_sj = sum_v exp(z_s - max_s) (z_s - z_j) for every j != s (the difference
// is taken element by element, so nearly equal sub-models lose no precision).
// TMEM is a ring of four 128-column slots: the u-th unit (one sub-model of one
// vocabulary tile, widest sub-model first) goes to slot u mod 4 and waits only
// for that slot's previous tile to be drained, so at M = 3 the next tile's
// widest unit runs during the epilogue (M = 2: full double buffering; M = 4:
// one tile at a time).  Roles: warp 8 TMA producer, warp 9 MMA issuer (even
// CTA), warps 0-7 epilogue (one thread per token and 64 columns).
#include <climits>

#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

struct EvalSmem {
  static constexpr uint32_t kA = 0;
  static constexpr uint32_t kB = kEvalStages * kEvalABytes;
  static constexpr uint32_t kX = kA;  // half-merge exchange, after the main loop only
  static constexpr uint32_t kBar = kB + kEvalStages * kEvalBBytes;
  static __device__ __forceinline__ uint32_t full(uint32_t b, int s) { return b + kBar + 8u * s; }
  static __device__ __forceinline__ uint32_t empty(uint32_t b, int s) {
    return b + kBar + 8u * (kEvalStages + s);
  }
  // tile j's accumulators are complete: accf(j mod 4); slot s drained: slote(s)
  static __device__ __forceinline__ uint32_t accf(uint32_t b, int j) {
    return b + kBar + 8u * (2 * kEvalStages + (j & 3));
  }
  static __device__ __forceinline__ uint32_t slote(uint32_t b, int s) {
    return b + kBar + 8u * (2 * kEvalStages + 4 + s);
  }
  static __device__ __forceinline__ uint32_t drain(uint32_t b) {
    return b + kBar + 8u * (2 * kEvalStages + 8);
  }
  static constexpr uint32_t kTmemSlot = kBar + 8u * (2 * kEvalStages + 9);
  static constexpr uint32_t kAbort = kTmemSlot + 4;
  static constexpr uint32_t kEnd = kAbort + 4;
};
static_assert(EvalSmem::kEnd + 1024 <= kEvalSmem, "eval shared memory map overflows");
static_assert(kMaxModels * kEvalBN <= 512, "all sub-models' tiles must fit in TMEM");

constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kDrainNs = 100000000ull;
constexpr int kD = 12;  // field offset of D_sj

// field index of D_sj (j != s) in the partial state
__host__ __device__ constexpr int dfield(int s, int j) { return kD + s * 3 + (j < s ? j : j - 1); }

template <bool kTF32>
__device__ __forceinline__ void eval_producer(const EvalParams& p, uint32_t base, int row0,
                                              uint32_t rank, int split, volatile int* abort_flag) {
  constexpr int KE = kTF32 ? 32 : 64;
  int stage = 0;
  uint32_t phase = 0, filled = 0, lastpar = 0;
  bool ok = true;
  for (int vt = split; ok && vt < p.nvt; vt += p.S) {
    for (int i = 0; ok && i < p.M; ++i) {
      const int m = p.order[i];
      for (int kb = 0; kb < p.nk[m]; ++kb) {
        if (!mbar_wait(EvalSmem::empty(base, stage), phase ^ 1u, abort_flag, p.status)) {
          ok = false;
          break;
        }
        if (rank == 0) mbar_arrive_expect_tx(EvalSmem::full(base, stage), 2 * (kEvalABytes + kEvalBBytes));
        const uint32_t fb = map_to_rank(EvalSmem::full(base, stage), 0);
        tma_load_2d_pair(base + EvalSmem::kA + stage * kEvalABytes, &p.mapH[m], fb, kb * KE, row0);
        tma_load_2d_pair(base + EvalSmem::kB + stage * kEvalBBytes, &p.mapW[m], fb, kb * KE,
                         vt * kEvalBN + static_cast<int>(rank) * kEvalBHalf);
        filled |= 1u << stage;
        lastpar = (lastpar & ~(1u << stage)) | (phase << stage);
        if (++stage == kEvalStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
  }
  if (!ok && filled) {
    if (rank == 0) {
      for (int s = 0; s < kEvalStages; ++s)
        if ((filled >> s) & 1u) mbar_wait_drain(EvalSmem::full(base, s), (lastpar >> s) & 1u, kDrainNs, p.status);
    } else {
      spin_ns(kDrainNs);
    }
  }
}

template <bool kTF32>
__device__ __forceinline__ void eval_mma(const EvalParams& p, uint32_t base, uint32_t tmem,
                                         int split, volatile int* abort_flag) {
  constexpr uint32_t kIdesc = make_idesc(2 * kHeadBM, kEvalBN, kTF32, false, false);
  int stage = 0;
  uint32_t phase = 0;
  int uses[4] = {0, 0, 0, 0};  // times each TMEM slot has been handed out
  bool ok = true;
  int j = 0;
  for (int vt = split; ok && vt < p.nvt; vt += p.S, ++j) {
    for (int i = 0; ok && i < p.M; ++i) {
      const int m = p.order[i];
      const int slot = (j * p.M + i) & 3;
      // the n-th use of a slot waits for its (n-1)-th drain
      if (uses[slot] > 0 &&
          !mbar_wait(EvalSmem::slote(base, slot), static_cast<uint32_t>(uses[slot] - 1) & 1u,
                     abort_flag, p.status)) {
        ok = false;
        break;
      }
      ++uses[slot];
      tc_fence_after();
      const uint32_t d = tmem + static_cast<uint32_t>(slot) * kEvalBN;
      for (int kb = 0; kb < p.nk[m]; ++kb) {
        if (!mbar_wait(EvalSmem::full(base, stage), phase, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = make_sdesc(base + EvalSmem::kA + stage * kEvalABytes, 16);
        const uint64_t bd = make_sdesc(base + EvalSmem::kB + stage * kEvalBBytes, 16);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_issue_pair<kTF32>(d, ad + 2u * kk, bd + 2u * kk, kIdesc, (kb | kk) != 0);
        mma_commit_pair(EvalSmem::empty(base, stage), 0x3);
        if (++stage == kEvalStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok) break;
    mma_commit_pair(EvalSmem::accf(base, j), 0x3);
  }
  mma_commit_pair(EvalSmem::drain(base), 0x1);
  mbar_wait_drain(EvalSmem::drain(base), 0, kDrainNs, p.status);
}

struct EvalState {
  float m[kMaxModels], s[kMaxModels];
  int am[kMaxModels];
  float d[kMaxModels][kMaxModels];
};

// One 32-column chunk of every sub-model's tile (z[s][i] = z_s at column col0 + i).
template <bool kMasked>
__device__ __forceinline__ void eval_chunk(const float (&z)[kMaxModels][32], int M, int nvalid,
                                           long long col0, float L1, EvalState& st) {
#pragma unroll
  for (int s = 0; s < kMaxModels; ++s) {
    if (s >= M) continue;
    float cmax = -INFINITY;
    int carg = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const bool ok = !kMasked || i < nvalid;
      if (ok && z[s][i] > cmax) {
        cmax = z[s][i];
        carg = i;
      }
    }
    if (cmax > st.m[s]) {
      st.am[s] = static_cast<int>(col0 + carg);
      const float f = st.m[s] == -INFINITY ? 0.f : fast_exp2((st.m[s] - cmax) * L1);
      st.s[s] *= f;
#pragma unroll
      for (int j = 0; j < kMaxModels; ++j) st.d[s][j] *= f;
      st.m[s] = cmax;
    }
    const float nb = -st.m[s] * L1;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const bool ok = !kMasked || i < nvalid;
      const float e = ok ? fast_exp2(fmaf(z[s][i], L1, nb)) : 0.f;
      st.s[s] += e;
#pragma unroll
      for (int j = 0; j < kMaxModels; ++j)
        if (j != s && j < M) st.d[s][j] = fmaf(e, z[s][i] - z[j][i], st.d[s][j]);
    }
  }
}

__device__ __forceinline__ float scale_to(float from, float to, float L1) {
  return from == -INFINITY ? 0.f : fast_exp2((from - to) * L1);
}

__device__ __forceinline__ void eval_epilogue(const EvalParams& p, uint32_t base, uint32_t tmem,
                                              float* xchg, int row_base, int split, int warp,
                                              int lane, volatile int* abort_flag) {
  const int quad = warp & 3, half = warp >> 2;
  const int r = quad * 32 + lane;
  const long long row = static_cast<long long>(row_base) + r;
  const uint32_t tl = tmem + (static_cast<uint32_t>(quad * 32) << 16) + static_cast<uint32_t>(half * 64);
  const int M = p.M;
  const float L1 = p.L1;
  EvalState st;
#pragma unroll
  for (int s = 0; s < kMaxModels; ++s) {
    st.m[s] = -INFINITY;
    st.s[s] = 0.f;
    st.am[s] = 0;
#pragma unroll
    for (int j = 0; j < kMaxModels; ++j) st.d[s][j] = 0.f;
  }
  float z[kMaxModels][32];
  int j = 0;
  for (int vt = split; vt < p.nvt; vt += p.S, ++j) {
    const bool ok = mbar_wait(EvalSmem::accf(base, j), static_cast<uint32_t>(j >> 2) & 1u,
                              abort_flag, p.status);
    if (!__all_sync(0xffffffffu, ok)) break;
    tc_fence_after();
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const long long col0 = static_cast<long long>(vt) * kEvalBN + half * 64 + c * 32;
      const int nvalid = static_cast<int>(max(0LL, min(32LL, p.V - col0)));
      if (nvalid == 0) continue;  // warp-uniform
#pragma unroll
      for (int s = 0; s < kMaxModels; ++s)
        if (s < M) {
          const uint32_t slot = static_cast<uint32_t>(j * M + p.pos[s]) & 3u;
          tmem_ld32(tl + slot * kEvalBN + static_cast<uint32_t>(c * 32), z[s]);
        }
      if (nvalid == 32)
        eval_chunk<false>(z, M, 32, col0, L1, st);
      else
        eval_chunk<true>(z, M, nvalid, col0, L1, st);
    }
    tc_fence_before();
    __syncwarp();
    if (lane == 0)
      for (int i = 0; i < M; ++i)
        mbar_arrive_remote(map_to_rank(EvalSmem::slote(base, (j * M + i) & 3), 0));
  }

  // the two column halves of a token combine through shared memory
  auto X = [&](int f) -> float& { return xchg[f * kHeadBM + r]; };
  if (half == 1) {
#pragma unroll
    for (int s = 0; s < kMaxModels; ++s) {
      X(s) = st.m[s];
      X(4 + s) = st.s[s];
      X(8 + s) = __int_as_float(st.am[s]);
#pragma unroll
      for (int j = 0; j < kMaxModels; ++j)
        if (j != s) X(dfield(s, j)) = st.d[s][j];
    }
  }
  named_bar_sync(1, kHeadEpiWarps * 32);
  if (half == 1 || row >= p.T) return;
  float* P = p.part + static_cast<long long>(split) * kEvalFields * p.T + row;
#pragma unroll
  for (int s = 0; s < kMaxModels; ++s) {
    if (s >= M) continue;
    const float m1 = X(s), mm = fmaxf(st.m[s], m1);
    const float fa = scale_to(st.m[s], mm, L1), fb = scale_to(m1, mm, L1);
    const int a1 = __float_as_int(X(8 + s));
    P[s * p.T] = mm;
    P[(4 + s) * p.T] = st.s[s] * fa + X(4 + s) * fb;
    P[(8 + s) * p.T] = __int_as_float(m1 > st.m[s] ? a1 : (st.m[s] > m1 ? st.am[s] : min(st.am[s], a1)));
#pragma unroll
    for (int j = 0; j < kMaxModels; ++j)
      if (j != s && j < M) P[dfield(s, j) * p.T] = st.d[s][j] * fa + X(dfield(s, j)) * fb;
  }
}

template <bool kTF32>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kHeadThreads, 1)
    eval_kernel(const __grid_constant__ EvalParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(gbase + EvalSmem::kAbort);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + EvalSmem::kTmemSlot);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  int tt, split;
  band_unit(static_cast<int>(blockIdx.x >> 1), p.ntt, p.S, p.band, tt, split);
  const int row_base = tt * 2 * kHeadBM + static_cast<int>(rank) * kHeadBM;

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int s = 0; s < kEvalStages; ++s) {
      mbar_init(EvalSmem::full(base, s), 1);
      mbar_init(EvalSmem::empty(base, s), 1);
    }
    for (int q = 0; q < 4; ++q) {
      mbar_init(EvalSmem::accf(base, q), 1);
      mbar_init(EvalSmem::slote(base, q), 2 * kHeadEpiWarps);
    }
    mbar_init(EvalSmem::drain(base), 1);
    fence_barrier_init();
  }
  if (warp == kHeadEpiWarps + 1) {
    tmem_alloc_pair(base + EvalSmem::kTmemSlot, kTmemCols);
    tmem_relinquish_pair();
  }
  if (warp == kHeadEpiWarps && lane == 0) {
    for (int m = 0; m < p.M; ++m) {
      tma_prefetch_desc(&p.mapH[m]);
      tma_prefetch_desc(&p.mapW[m]);
    }
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp >= kHeadEpiWarps) {
    regs_decrease<kHeadCtlRegs>();
    if (warp == kHeadEpiWarps) {
      if (lane == 0) eval_producer<kTF32>(p, base, row_base, rank, split, abort_flag);
    } else if (warp == kHeadEpiWarps + 1) {
      if (lane == 0 && rank == 0) eval_mma<kTF32>(p, base, tmem, split, abort_flag);
      __syncwarp();
    }
  } else {
    regs_increase<kHeadEpiRegs>();
    eval_epilogue(p, base, tmem, reinterpret_cast<float*>(gbase + EvalSmem::kX), row_base, split,
                  warp, lane, abort_flag);
  }

  tc_fence_before();
  cluster_sync();
  if (warp == kHeadEpiWarps + 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------------ merge
__device__ __forceinline__ double block_sum(double v, double* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) sh[w] = v;
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0)
    for (int i = 0; i < static_cast<int>(blockDim.x >> 5); ++i) s += sh[i];
  return s;
}

constexpr int kEvalMergeThreads = 128;

__global__ void __launch_bounds__(kEvalMergeThreads)
    eval_merge_kernel(const __grid_constant__ EvalMergeParams p) {
  __shared__ double sh[kEvalMergeThreads / 32];
  const long long t = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  const int M = p.M;
  float kl[kMaxModels][kMaxModels] = {};
  int am[kMaxModels] = {};
  bool valid = false;
  if (t < p.T) {
    const float L1 = 1.4426950408889634f;
    const long long PS = static_cast<long long>(kEvalFields) * p.T;
    const float* P = p.part + t;
    float lse[kMaxModels], S[kMaxModels], D[kMaxModels][kMaxModels];
    for (int s = 0; s < M; ++s) {
      float mm = -INFINITY;
      for (int k = 0; k < p.nparts; ++k) mm = fmaxf(mm, P[k * PS + s * p.T]);
      float sum = 0.f;
      int a = INT_MAX;
      for (int j = 0; j < M; ++j) D[s][j] = 0.f;
      for (int k = 0; k < p.nparts; ++k) {
        const float* Q = P + k * PS;
        const float mk = Q[s * p.T];
        if (mk == -INFINITY) continue;
        const float f = exp2f((mk - mm) * L1);
        sum += Q[(4 + s) * p.T] * f;
        for (int j = 0; j < M; ++j)
          if (j != s) D[s][j] += Q[dfield(s, j) * p.T] * f;
        if (mk == mm) a = min(a, __float_as_int(Q[(8 + s) * p.T]));
      }
      S[s] = sum;
      lse[s] = mm + logf(sum);
      am[s] = a;
    }
    for (int s = 0; s < M; ++s)
      for (int j = 0; j < M; ++j)
        kl[s][j] = (s == j) ? 0.f : D[s][j] / S[s] - (lse[s] - lse[j]);
    const int y = p.y ? p.y[t] : 0;
    if (p.y && y >= p.V) atomicOr(p.status, kStatusBadTarget);
    valid = !p.y || (y >= 0 && y < p.V);
    for (int s = 0; s < M; ++s) {
      for (int j = 0; j < M; ++j) p.tok_kl[(static_cast<long long>(s) * M + j) * p.T + t] = kl[s][j];
      if (p.argmax) p.argmax[static_cast<long long>(s) * p.T + t] = am[s];
    }
  }
  double* out = p.block_acc + static_cast<long long>(blockIdx.x) * 2 * kMaxModels * kMaxModels;
  for (int s = 0; s < M; ++s) {
    for (int j = 0; j < M; ++j) {
      const double a = block_sum(valid ? static_cast<double>(kl[s][j]) : 0.0, sh);
      const double b = block_sum(valid && am[s] == am[j] ? 1.0 : 0.0, sh);
      if (threadIdx.x == 0) {
        out[s * M + j] = a;
        out[kMaxModels * kMaxModels + s * M + j] = b;
      }
    }
  }
  const double c = block_sum(valid ? 1.0 : 0.0, sh);
  if (threadIdx.x == 0) p.block_cnt[blockIdx.x] = static_cast<long long>(c);
}

constexpr int kEvalFinalThreads = 256;

__global__ void __launch_bounds__(kEvalFinalThreads)
    eval_final_kernel(const double* __restrict__ acc, const long long* __restrict__ cnt, int n,
                      int M, float* pair_stats) {
  __shared__ double sh[kEvalFinalThreads / 32];
  double c = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) c += static_cast<double>(cnt[i]);
  const double C = block_sum(c, sh);
  __shared__ double Cs;
  if (threadIdx.x == 0) Cs = C;
  for (int q = 0; q < 2; ++q) {
    for (int e = 0; e < M * M; ++e) {
      double s = 0.0;
      for (int i = threadIdx.x; i < n; i += blockDim.x)
        s += acc[static_cast<long long>(i) * 2 * kMaxModels * kMaxModels + q * kMaxModels * kMaxModels + e];
      const double S = block_sum(s, sh);
      if (threadIdx.x == 0) pair_stats[q * M * M + e] = Cs > 0.0 ? static_cast<float>(S / Cs) : 0.f;
    }
  }
}

}  // namespace

cudaError_t launch_eval(const EvalParams& p, bool tf32, cudaStream_t s) {
  const int grid = 2 * p.ntt * p.S;
  if (grid <= 0) return cudaSuccess;
  if (tf32)
    eval_kernel<true><<<grid, kHeadThreads, kEvalSmem, s>>>(p);
  else
    eval_kernel<false><<<grid, kHeadThreads, kEvalSmem, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_eval_merge(const EvalMergeParams& p, int blocks, cudaStream_t s) {
  if (blocks <= 0) return cudaSuccess;
  eval_merge_kernel<<<blocks, kEvalMergeThreads, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_eval_final(const double* block_acc, const long long* block_cnt, int nblocks,
                              int M, float* pair_stats, cudaStream_t s) {
  eval_final_kernel<<<1, kEvalFinalThreads, 0, s>>>(block_acc, block_cnt, nblocks, M, pair_stats);
  return cudaGetLastError();
}

cudaError_t setup_eval_kernels() {
  cudaError_t e;
#define MLS_SET(TF)                                                                           \
  e = cudaFuncSetAttribute(eval_kernel<TF>, cudaFuncAttributeMaxDynamicSharedMemorySize,      \
                           kEvalSmem);                                                        \
  if (e != cudaSuccess) return e;                                                             \
  {                                                                                           \
    cudaFuncAttributes fa;                                                                    \
    e = cudaFuncGetAttributes(&fa, eval_kernel<TF>);                                          \
    if (e != cudaSuccess) return e;                                                           \
    if (fa.maxThreadsPerBlock < kHeadThreads || fa.numRegs != kHeadLaunchRegs)                \
      return cudaErrorLaunchOutOfResources;                                                   \
  }
  MLS_SET(true)
  MLS_SET(false)
#undef MLS_SET
  return cudaSuccess;
}

}  // namespace mls
