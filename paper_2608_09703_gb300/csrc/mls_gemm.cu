// Gradient GEMMs of the backward pass, on tcgen05 tensor cores:
//   dW_m[v, :] = sum_t G_m[t, v] H_m[t, :]     A = G_m viewed M-major (M = v), B = H_m N-major
//   dH_m[t, :] = sum_v G_m[t, v] W_m[v, :]     A = G_m K-major (K = v),       B = W_m N-major
// where G_m = dL/dz_m is the bf16 (fp32 for fp32 inputs) gradient tile written
// by the backward head kernel.  For bf16 both products read the row-major
// tensors in place: the shared-memory descriptors say which dimension is
// contiguous, so no transposed copy of G, H or W is made.  The tf32 MMA is
// only used with K-major operands here, so fp32 inputs go through transposed
// copies (G^T, H^T, W^T) instead.
//
// CTA pairs (clusters of 2) own 256x256 output tiles: each CTA loads the 128
// rows of A and the 128 rows of B that are its half, the even CTA issues
// 256x256xK pair MMAs (cta_group::2) and each CTA drains its 128 accumulator
// rows.  Persistent pairs walk a list of units over up to eight problems (dW
// and dH of each sub-model); a unit is one output tile, or for a wide problem
// two adjacent column tiles that share each stage's A tile and use both TMEM
// accumulators (no epilogue overlap, so only long reductions are made wide):
//   warp 4    TMA producer (each CTA its own halves; both CTAs' loads complete
//             on the even CTA's barrier, which expects the bytes of both)
//   warp 5    MMA issuer (even CTA)
//   warps 0-3 epilogue (each CTA its 128 rows)
#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

struct GemmSmem {
  static constexpr uint32_t kA = 0;
  static constexpr uint32_t kB = kGemmStages * kGemmABytes;
  static constexpr uint32_t kBar = kB + kGemmStages * kGemmBBytes;
  // full (even CTA): both CTAs' loads landed; empty: the pair's MMAs are done
  // with the stage; accf/acce: accumulator full/empty.
  static __device__ __forceinline__ uint32_t full(uint32_t b, int s) { return b + kBar + 8u * s; }
  static __device__ __forceinline__ uint32_t empty(uint32_t b, int s) {
    return b + kBar + 8u * (kGemmStages + s);
  }
  static __device__ __forceinline__ uint32_t accf(uint32_t b, uint32_t a) {
    return b + kBar + 8u * (2 * kGemmStages + a);
  }
  static __device__ __forceinline__ uint32_t acce(uint32_t b, uint32_t a) {
    return b + kBar + 8u * (2 * kGemmStages + 2 + a);
  }
  static __device__ __forceinline__ uint32_t drain(uint32_t b) {
    return b + kBar + 8u * (2 * kGemmStages + 4);
  }
  // Wide units: stage s holds A | B0 | B1 at s * kWideStage, over the memory of
  // the plain stages; wfull / wempty are its barriers.
  static constexpr uint32_t kWideStage = kGemmABytes + 2 * kGemmBBytes;
  static __device__ __forceinline__ uint32_t wfull(uint32_t b, int s) {
    return b + kBar + 8u * (2 * kGemmStages + 5 + s);
  }
  static __device__ __forceinline__ uint32_t wempty(uint32_t b, int s) {
    return b + kBar + 8u * (2 * kGemmStages + 5 + kGemmWideStages + s);
  }
  static constexpr uint32_t kTmemSlot = kBar + 8u * (2 * kGemmStages + 5 + 2 * kGemmWideStages);
  static constexpr uint32_t kAbort = kTmemSlot + 4;
  static constexpr uint32_t kEnd = kAbort + 4;
  // kEpiSoftmax output staging: per epilogue warp two 32 x 32 fp32 chunks
  // (128B-swizzled) written out by TMA stores.  It lies in the slack past the
  // operand stages, which only the MN-major (plain-epilogue) GEMMs over-read.
  static constexpr uint32_t kChunk = 32 * 32 * 4;
  static constexpr uint32_t kStaging = (kEnd + 1023u) & ~1023u;
};
static_assert(GemmSmem::kEnd + 1024 <= kGemmSmem, "gemm shared memory map overflows");
static_assert(kGemmWideStages * GemmSmem::kWideStage <= GemmSmem::kBar,
              "wide stages must fit in the plain stages' memory");
static_assert(GemmSmem::kWideStage % 1024 == 0, "wide stages must stay 1024-byte aligned");
static_assert(GemmSmem::kStaging + kGemmEpiWarps * 2 * GemmSmem::kChunk + 1023 <= kGemmSmem,
              "gemm output staging overflows");

constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kDrainNs = 100000000ull;
constexpr int kPairM = 2 * kGemmBM;  // output rows of a pair tile

struct UnitCoord {
  int prob, tm, tn, nt;  // problem, tile row, first tile column, tiles (1 or 2)
};

// The j-th unit of this pair, or -1 when it has no more.
__device__ __forceinline__ int pair_unit(const GemmParams& p, int pair, int npairs, int j) {
  if (!p.two_class) {
    const int t = pair + j * npairs;
    return t < p.total_tiles ? t : -1;
  }
  const int r = p.n_long % npairs;
  const int nl = p.n_long / npairs + (pair < r ? 1 : 0);
  if (j < nl) return pair + j * npairs;
  j -= nl;
  const int n_short = p.total_tiles - p.n_long;
  if (pair >= r) {
    if (j < p.catchup) return p.n_long + (pair - r) + j * (npairs - r);
    j -= p.catchup;
  }
  const int s = p.catchup * (npairs - r) + pair + j * npairs;
  return s < n_short ? p.n_long + s : -1;
}

// A is MN-major for this problem.
template <int kAMode>
__device__ __forceinline__ bool a_mn_of(const GemmProblem& pr) {
  return kAMode == 2 ? pr.a_mn != 0 : kAMode == 1;
}

// Wide units exist only in the launch that mixes problems (launch_gemm_mixed).
template <int kAMode>
__device__ __forceinline__ bool wide_of(const GemmProblem& pr) {
  return kAMode == 2 && pr.wide != 0;
}

template <int kAMode>
__device__ __forceinline__ UnitCoord decode_unit(const GemmParams& p, int u) {
  int i = 0;
  while (i + 1 < p.nprob && u >= p.prob[i + 1].tile_begin) ++i;
  const GemmProblem& pr = p.prob[i];
  const int local = u - pr.tile_begin;
  if (pr.m_fast) return {i, local % pr.tiles_m, local / pr.tiles_m, 1};
  if (wide_of<kAMode>(pr)) {
    const int un = (pr.tiles_n + 1) >> 1;
    const int tn = (local % un) * 2;
    return {i, local / un, tn, pr.tiles_n - tn < 2 ? 1 : 2};
  }
  return {i, local / pr.tiles_n, local % pr.tiles_n, 1};
}

// This CTA's loads: its 128 rows of A and its 128 rows of B (of both column
// tiles in a wide unit) for every k-block.
template <bool kTF32, int kAMode, bool kBMN>
__device__ __forceinline__ void gemm_producer(const GemmParams& p, uint32_t base, uint32_t rank,
                                              volatile int* abort_flag) {
  constexpr int KE = kTF32 ? 32 : 64;  // elements per 128-byte row
  constexpr uint32_t kBox = KE * 128;  // bytes of one MN-major box {KE, KE}
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  // plain ring (kGemmStages) and wide ring (kGemmWideStages) over the same memory
  int stage = 0, wstage = 0;
  uint32_t phase = 0, filled = 0, lastpar = 0;
  uint32_t wphase = 0, wfilled = 0, wlastpar = 0;
  int layout = -1;  // ring the stages were last filled in: 0 plain, 1 wide
  bool ok = true;
  int u;
  for (int j = 0; ok && (u = pair_unit(p, pair, npairs, j)) >= 0; ++j) {
    const UnitCoord uc = decode_unit<kAMode>(p, u);
    const GemmProblem& pr = p.prob[uc.prob];
    MLS_CHECK(p.status, u < p.total_tiles && uc.prob < p.nprob && pr.a_map < kGemmMaxProblems &&
                            static_cast<long long>(uc.tm) * kPairM < pr.Mrows &&
                            static_cast<long long>(uc.tn + uc.nt - 1) * kGemmBN < pr.Ncols);
    const bool amn = a_mn_of<kAMode>(pr);
    const bool wide = wide_of<kAMode>(pr);
    // Before one ring's memory is refilled in the other layout, every stage
    // filled in the old layout must have been consumed by the MMAs.
    if (layout == (wide ? 0 : 1)) {
      for (int s = 0; ok && s < (wide ? kGemmStages : kGemmWideStages); ++s) {
        const uint32_t f = wide ? filled : wfilled, lp = wide ? lastpar : wlastpar;
        if ((f >> s) & 1u)
          ok = mbar_wait(wide ? GemmSmem::empty(base, s) : GemmSmem::wempty(base, s), (lp >> s) & 1u,
                         abort_flag, p.status);
      }
      if (!ok) break;
    }
    layout = wide ? 1 : 0;
    const CUtensorMap* ma = &p.mapA[pr.a_map];
    const CUtensorMap* mb = &p.mapB[pr.b_map];
    const int nkb = (pr.K + KE - 1) / KE;
    const int m0 = pr.a_m0 + uc.tm * kPairM + static_cast<int>(rank) * kGemmBM;
    const int n0 = pr.b_n0 + uc.tn * kGemmBN + static_cast<int>(rank) * kGemmBHalf;
    for (int kb = 0; kb < nkb; ++kb) {
      const uint32_t empty_bar = wide ? GemmSmem::wempty(base, wstage) : GemmSmem::empty(base, stage);
      if (!mbar_wait(empty_bar, (wide ? wphase : phase) ^ 1u, abort_flag, p.status)) {
        ok = false;
        break;
      }
      const uint32_t full_bar = wide ? GemmSmem::wfull(base, wstage) : GemmSmem::full(base, stage);
      const uint32_t fb = map_to_rank(full_bar, 0);
      if (rank == 0)
        mbar_arrive_expect_tx(full_bar, 2 * (kGemmABytes + static_cast<uint32_t>(uc.nt) * kGemmBBytes));
      const uint32_t sa = wide ? base + wstage * GemmSmem::kWideStage : base + GemmSmem::kA + stage * kGemmABytes;
      const uint32_t sb = wide ? sa + kGemmABytes : base + GemmSmem::kB + stage * kGemmBBytes;
      const int ka = pr.a_k0 + kb * KE, kbb = pr.b_k0 + kb * KE;
      if (amn) {
#pragma unroll
        for (int q = 0; q < kGemmBM / KE; ++q) tma_load_2d_pair(sa + q * kBox, ma, fb, m0 + q * KE, ka);
      } else {
        tma_load_2d_pair(sa, ma, fb, ka, m0);
      }
      for (int t = 0; t < uc.nt; ++t) {
        const uint32_t sbt = sb + static_cast<uint32_t>(t) * kGemmBBytes;
        const int n0t = n0 + t * kGemmBN;
        if (kBMN) {
#pragma unroll
          for (int q = 0; q < kGemmBHalf / KE; ++q) tma_load_2d_pair(sbt + q * kBox, mb, fb, n0t + q * KE, kbb);
        } else {
          tma_load_2d_pair(sbt, mb, fb, kbb, n0t);
        }
      }
      if (wide) {
        wfilled |= 1u << wstage;
        wlastpar = (wlastpar & ~(1u << wstage)) | (wphase << wstage);
        if (++wstage == kGemmWideStages) {
          wstage = 0;
          wphase ^= 1u;
        }
      } else {
        filled |= 1u << stage;
        lastpar = (lastpar & ~(1u << stage)) | (phase << stage);
        if (++stage == kGemmStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
  }
  if (!ok && (filled | wfilled)) {
    // Loads already issued must land before this CTA's shared memory goes away.
    // The even CTA can watch its barriers; the odd CTA's loads are counted on
    // the even CTA's barriers, so it waits out a bound no TMA load approaches.
    if (rank == 0) {
      for (int s = 0; s < kGemmStages; ++s)
        if ((filled >> s) & 1u)
          mbar_wait_drain(GemmSmem::full(base, s), (lastpar >> s) & 1u, kDrainNs, p.status);
      for (int s = 0; s < kGemmWideStages; ++s)
        if ((wfilled >> s) & 1u)
          mbar_wait_drain(GemmSmem::wfull(base, s), (wlastpar >> s) & 1u, kDrainNs, p.status);
    } else {
      spin_ns(kDrainNs);
    }
  }
}

// Tile i of this pair (counted over its units) accumulates in TMEM
// accumulator i & 1, whose (i >> 1)-th use it is.
template <bool kTF32, int kAMode, bool kBMN>
__device__ __forceinline__ void gemm_mma(const GemmParams& p, uint32_t base, uint32_t tmem,
                                         volatile int* abort_flag) {
  constexpr int KE = kTF32 ? 32 : 64;
  constexpr uint32_t kBox = KE * 128;
  // Advance per MMA (32 bytes of K): along a 128-byte row for K-major
  // operands, by (32 / element size) rows of 128 bytes for MN-major ones.
  constexpr uint32_t kStepK = 32u >> 4;
  constexpr uint32_t kStepMN = ((32u / (kTF32 ? 4u : 2u)) * 128u) >> 4;
  constexpr uint16_t kBoth = 0x3;
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  int stage = 0, wstage = 0;
  uint32_t phase = 0, wphase = 0, tiles = 0;
  bool ok = true;
  int u;
  for (int j = 0; ok && (u = pair_unit(p, pair, npairs, j)) >= 0; ++j) {
    const UnitCoord uc = decode_unit<kAMode>(p, u);
    const GemmProblem& pr = p.prob[uc.prob];
    const int nkb = (pr.K + KE - 1) / KE;
    const bool amn = a_mn_of<kAMode>(pr);
    const bool wide = wide_of<kAMode>(pr);
    const uint32_t idesc = make_idesc(kPairM, kGemmBN, kTF32, amn, kBMN);
    for (int t = 0; ok && t < uc.nt; ++t) {
      const uint32_t i = tiles + static_cast<uint32_t>(t);
      ok = mbar_wait(GemmSmem::acce(base, i & 1u), ((i >> 1) & 1u) ^ 1u, abort_flag, p.status);
    }
    if (!ok) break;
    tc_fence_after();
    const uint32_t d0 = tmem + (tiles & 1u) * kGemmBN, d1 = tmem + ((tiles + 1u) & 1u) * kGemmBN;
    for (int kb = 0; kb < nkb; ++kb) {
      const uint32_t full_bar = wide ? GemmSmem::wfull(base, wstage) : GemmSmem::full(base, stage);
      if (!mbar_wait(full_bar, wide ? wphase : phase, abort_flag, p.status)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t sa = wide ? base + wstage * GemmSmem::kWideStage : base + GemmSmem::kA + stage * kGemmABytes;
      const uint32_t sb = wide ? sa + kGemmABytes : base + GemmSmem::kB + stage * kGemmBBytes;
      const uint64_t ad = make_sdesc(sa, amn ? kBox : 16u);
      const uint64_t bd = make_sdesc(sb, kBMN ? kBox : 16u);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        mma_issue_pair<kTF32>(d0, ad + kk * (amn ? kStepMN : kStepK),
                              bd + kk * (kBMN ? kStepMN : kStepK), idesc, (kb | kk) != 0);
      if (uc.nt == 2) {
        const uint64_t bd1 = make_sdesc(sb + kGemmBBytes, kBMN ? kBox : 16u);  // second column tile
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_issue_pair<kTF32>(d1, ad + kk * (amn ? kStepMN : kStepK),
                                bd1 + kk * (kBMN ? kStepMN : kStepK), idesc, (kb | kk) != 0);
      }
      if (wide) {
        mma_commit_pair(GemmSmem::wempty(base, wstage), kBoth);
        if (++wstage == kGemmWideStages) {
          wstage = 0;
          wphase ^= 1u;
        }
      } else {
        mma_commit_pair(GemmSmem::empty(base, stage), kBoth);
        if (++stage == kGemmStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok) break;
    for (int t = 0; t < uc.nt; ++t) mma_commit_pair(GemmSmem::accf(base, (tiles + t) & 1u), kBoth);
    tiles += static_cast<uint32_t>(uc.nt);
  }
  mma_commit_pair(GemmSmem::drain(base), 0x1);
  mbar_wait_drain(GemmSmem::drain(base), 0, kDrainNs, p.status);
}

// Largest of 32 values, as a tree (depth 5, not a 32-step chain).
__device__ __forceinline__ float max32(const float (&v)[32]) {
  float m[16];
#pragma unroll
  for (int i = 0; i < 16; ++i) m[i] = fmaxf(v[i], v[i + 16]);
#pragma unroll
  for (int w = 8; w > 0; w >>= 1)
#pragma unroll
    for (int i = 0; i < w; ++i) m[i] = fmaxf(m[i], m[i + w]);
  return m[0];
}

// Row statistics epilogues (kEpiSoftmax, kEpiArgmax) of one 128 x kGemmBN
// accumulator tile: each lane owns one row, and `ncols` of its columns lie
// inside C.  kEpiArgmax reads the row's accumulators once for the maximum and
// its first column.  kEpiSoftmax reads them once for the maximum m_t and again
// to store e = 2^((z - m_t) scale) and sum it.
// Each epilogue warp runs alone on its SM sub-partition, so latency is not
// hidden by other warps; the softmax passes avoid long dependent chains (the
// maximum is a tree, the sum four interleaved partial sums).  Its cost must
// stay under the MMAs of the next tile, ~8.4k cycles for a K = 1024 tile; with
// 32-step chains it took ~16k cycles.
__device__ __noinline__ void epilogue_stats(const GemmProblem& pr, const CUtensorMap* mapC,
                                            uint32_t stage, uint32_t& count, uint32_t tacc,
                                            int tn, long long row, bool row_ok, int row0,
                                            int lane) {
  float v[32];
  float mt = -INFINITY;
  const int col0 = tn * kGemmBN;
  const int ncols = pr.Ncols - col0;  // >= 1: a tile starts inside C
  float* srow = pr.stats + (row_ok ? row : 0) * pr.stats_ld + 2 * tn;
  if (pr.epi == kEpiArgmax) {
    int mi = col0;
#pragma unroll 1
    for (int c = 0; c < kGemmBN / 32; ++c) {
      tmem_ld32(tacc + c * 32, v);
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (c * 32 + i < ncols && v[i] > mt) {
          mt = v[i];
          mi = col0 + c * 32 + i;
        }
    }
    if (row_ok) {
      srow[0] = mt;
      srow[1] = __int_as_float(mi);
    }
    return;
  }
  const int nchunks = ncols < kGemmBN ? (ncols + 31) / 32 : kGemmBN / 32;
#pragma unroll 1
  for (int c = 0; c < nchunks; ++c) {
    tmem_ld32(tacc + c * 32, v);
    if (c * 32 + 32 > ncols) {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (c * 32 + i >= ncols) v[i] = -INFINITY;
    }
    mt = fmaxf(mt, max32(v));
  }
  // Two chunks (both staging buffers) per round: one proxy fence and one
  // bulk group for 32 rows x 64 columns.
  float st = 0.f;
#pragma unroll 1
  for (int c = 0; c < nchunks; c += 2) {
    float w[2][32];
    tmem_ld32(tacc + c * 32, w[0]);
    if (c + 1 < nchunks) tmem_ld32(tacc + c * 32 + 32, w[1]);
    float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int cc = (c + h) * 32;
      if (cc + 32 <= ncols) {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          w[h][i] = fast_exp2((w[h][i] - mt) * pr.epi_scale);
          s4[i & 3] += w[h][i];
        }
      } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          w[h][i] = cc + i < ncols ? fast_exp2((w[h][i] - mt) * pr.epi_scale) : 0.f;
          s4[i & 3] += w[h][i];
        }
      }
    }
    st += (s4[0] + s4[1]) + (s4[2] + s4[3]);
    // 32 rows x 32 columns per buffer through shared memory; the TMA store
    // drops rows and columns outside C.
    if (lane == 0) bulk_wait_read<0>();  // the previous round's stores have read both buffers
    __syncwarp();
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const uint32_t rowaddr = stage + h * GemmSmem::kChunk + lane * 128;
#pragma unroll
      for (int j = 0; j < 8; ++j)
        st_shared_v4(rowaddr + ((j ^ (lane & 7)) << 4), __float_as_uint(w[h][4 * j]),
                     __float_as_uint(w[h][4 * j + 1]), __float_as_uint(w[h][4 * j + 2]),
                     __float_as_uint(w[h][4 * j + 3]));
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(mapC, stage, col0 + c * 32, row0);
      if (c + 1 < nchunks) tma_store_2d(mapC, stage + GemmSmem::kChunk, col0 + c * 32 + 32, row0);
      bulk_commit();
    }
    ++count;
  }
  if (row_ok) {
    srow[0] = mt;
    srow[1] = st;
  }
}

// kStats: the launch may hold problems with a statistics epilogue (only the
// verify step's logits GEMM); without it epilogue_stats is not in the kernel,
// which keeps the training GEMMs at 64 registers instead of 119.
template <int kAMode, bool kStats>
__device__ __forceinline__ void gemm_epilogue(const GemmParams& p, uint32_t base, uint32_t tmem,
                                              uint32_t rank, int warp, int lane,
                                              volatile int* abort_flag) {
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  uint32_t tiles = 0, stores = 0;
  const uint32_t tl = tmem + (static_cast<uint32_t>(warp * 32) << 16);
  const uint32_t stage = base + GemmSmem::kStaging + static_cast<uint32_t>(warp) * 2 * GemmSmem::kChunk;
  bool aborted = false;
  int u;
  for (int j = 0; !aborted && (u = pair_unit(p, pair, npairs, j)) >= 0; ++j) {
    const UnitCoord uc = decode_unit<kAMode>(p, u);
    const GemmProblem& pr = p.prob[uc.prob];
    for (int t = 0; t < uc.nt; ++t, ++tiles) {
      const uint32_t acc = tiles & 1u;
      const int tn = uc.tn + t;
      const bool ok = mbar_wait(GemmSmem::accf(base, acc), (tiles >> 1) & 1u, abort_flag, p.status);
      if (!__all_sync(0xffffffffu, ok)) {
        aborted = true;
        break;
      }
      tc_fence_after();
      const long long row = static_cast<long long>(uc.tm) * kPairM + rank * kGemmBM + warp * 32 + lane;
      const bool row_ok = row < pr.Mrows;
      float v[32];
      if (kStats && pr.epi != kEpiPlain) {
        const int row0 = uc.tm * kPairM + static_cast<int>(rank) * kGemmBM + warp * 32;
        epilogue_stats(pr, &p.mapC[uc.prob], stage, stores, tl + acc * kGemmBN, tn, row, row_ok,
                       row0, lane);
      } else {
        float* crow = pr.C + (row_ok ? row : 0) * pr.ldc;
#pragma unroll 1
        for (int c = 0; c < kGemmBN / 32; ++c) {
          tmem_ld32(tl + acc * kGemmBN + c * 32, v);
          const int col = tn * kGemmBN + c * 32;
          if (row_ok && col < pr.Ncols) {
            float* dst = crow + col;
            if (col + 32 <= pr.Ncols) {
              float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                float4 o = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                if (pr.accumulate) {
                  const float4 c4 = d4[i];
                  o.x += c4.x;
                  o.y += c4.y;
                  o.z += c4.z;
                  o.w += c4.w;
                }
                d4[i] = o;
              }
            } else {
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (col + i < pr.Ncols) dst[i] = pr.accumulate ? dst[i] + v[i] : v[i];
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(map_to_rank(GemmSmem::acce(base, acc), 0));
    }
  }
  if (stores && lane == 0) bulk_wait_all();  // staging must outlive the stores reading it
}

template <bool kTF32, int kAMode, bool kBMN, bool kStats>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
    gemm_kernel(const __grid_constant__ GemmParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(gbase + GemmSmem::kAbort);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + GemmSmem::kTmemSlot);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int s = 0; s < kGemmStages; ++s) {
      mbar_init(GemmSmem::full(base, s), 1);
      mbar_init(GemmSmem::empty(base, s), 1);
    }
    for (int s = 0; s < kGemmWideStages; ++s) {
      mbar_init(GemmSmem::wfull(base, s), 1);
      mbar_init(GemmSmem::wempty(base, s), 1);
    }
    for (uint32_t a = 0; a < 2; ++a) {
      mbar_init(GemmSmem::accf(base, a), 1);
      mbar_init(GemmSmem::acce(base, a), 2 * kGemmEpiWarps);
    }
    mbar_init(GemmSmem::drain(base), 1);
    fence_barrier_init();
  }
  if (warp == kGemmEpiWarps + 1) {
    tmem_alloc_pair(base + GemmSmem::kTmemSlot, kTmemCols);
    tmem_relinquish_pair();
  }
  if (warp == kGemmEpiWarps && lane == 0) {
    for (int i = 0; i < p.nprob; ++i) {
      tma_prefetch_desc(&p.mapA[p.prob[i].a_map]);
      tma_prefetch_desc(&p.mapB[p.prob[i].b_map]);
    }
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == kGemmEpiWarps) {
    if (lane == 0) gemm_producer<kTF32, kAMode, kBMN>(p, base, rank, abort_flag);
  } else if (warp == kGemmEpiWarps + 1) {
    if (lane == 0 && rank == 0) gemm_mma<kTF32, kAMode, kBMN>(p, base, tmem, abort_flag);
    __syncwarp();
  } else {
    gemm_epilogue<kAMode, kStats>(p, base, tmem, rank, warp, lane, abort_flag);
  }

  tc_fence_before();
  cluster_sync();
  if (warp == kGemmEpiWarps + 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kTmemCols);
  }
}

template <int kAMode, bool kBMN, bool kStats>
cudaError_t launch(const GemmParams& p, bool tf32, int grid, cudaStream_t s) {
  if (p.total_tiles <= 0 || grid <= 0) return cudaSuccess;
  if (tf32)
    gemm_kernel<true, kAMode, kBMN, kStats><<<grid, kGemmThreads, kGemmSmem, s>>>(p);
  else
    gemm_kernel<false, kAMode, kBMN, kStats><<<grid, kGemmThreads, kGemmSmem, s>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_kk(const GemmParams& p, bool tf32, int grid, cudaStream_t s) {
  return launch<0, false, false>(p, tf32, grid, s);
}
cudaError_t launch_gemm_stats(const GemmParams& p, bool tf32, int grid, cudaStream_t s) {
  return launch<0, false, true>(p, tf32, grid, s);
}
cudaError_t launch_gemm_mixed(const GemmParams& p, int grid, cudaStream_t s) {
  if (p.total_tiles <= 0 || grid <= 0) return cudaSuccess;
  gemm_kernel<false, 2, true, false><<<grid, kGemmThreads, kGemmSmem, s>>>(p);
  return cudaGetLastError();
}

// How many CTA pairs of the GEMM kernel can be resident at once (GPCs with an
// odd number of free SMs host one CTA fewer than a pair needs).
int gemm_max_active_pairs() {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * 1024);
  cfg.blockDim = dim3(kGemmThreads);
  cfg.dynamicSmemBytes = kGemmSmem;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, gemm_kernel<false, 2, true, false>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t setup_gemm_kernels() {
  cudaError_t e;
#define MLS_SET(TF, AM, BM, ST)                                                                 \
  e = cudaFuncSetAttribute(gemm_kernel<TF, AM, BM, ST>,                                         \
                           cudaFuncAttributeMaxDynamicSharedMemorySize, kGemmSmem);             \
  if (e != cudaSuccess) return e;                                                               \
  {                                                                                             \
    cudaFuncAttributes fa;                                                                      \
    e = cudaFuncGetAttributes(&fa, gemm_kernel<TF, AM, BM, ST>);                                \
    if (e != cudaSuccess) return e;                                                             \
    if (fa.maxThreadsPerBlock < kGemmThreads) return cudaErrorLaunchOutOfResources;             \
  }
  MLS_SET(true, 0, false, false)
  MLS_SET(false, 0, false, false)
  MLS_SET(true, 0, false, true)
  MLS_SET(false, 0, false, true)
  MLS_SET(false, 2, true, false)
#undef MLS_SET
  return cudaSuccess;
}

}  // namespace mls
