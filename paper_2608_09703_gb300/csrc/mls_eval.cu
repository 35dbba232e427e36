// Forward-only evaluation metrics between the sub-models of a suite
// (paper Sec. 3.2.2: pairwise KL divergence and top-1 agreement; App. A plots
// KL(p_student || p_teacher)).  For every token and ordered pair (s, j):
//   KL(p_s || p_j) = E_{p_s}[z_s - z_j] - (lse_s - lse_j)
// with p = softmax(z) at temperature 1.  The logits are never stored.
//
// A CTA pair owns 256 tokens and a strided set of vocabulary tiles of
// N = eval_tile_cols(M) columns (256 for M <= 3, 128 for M = 4).  For each tile
// the even CTA issues pair MMAs (cta_group::2, 256 x N x K) for every
// sub-model, widest first (unit position q holds sub-model order[q]); the
// epilogue accumulates, per sub-model s, the running max, sum_v exp(z_s - max_s)
// and D_sj = sum_v exp(z_s - max_s) (z_s - z_j) for every j != s (the
// difference is taken element by element, so nearly equal sub-models lose no
// precision).  The epilogue first copies the widest sub-model's tile into
// registers and releases its TMEM columns, so the next MMAs run while it reads
// the other sub-models from TMEM.  Two TMEM schedules:
//   - all resident (M = 1, 2, 4): unit q in columns [qN, (q+1)N), M N <= 512;
//     the next tile's widest unit runs under the rest of the epilogue;
//   - slots (M = 3): the two narrower units in two 256-column slots; the
//     epilogue passes over them pair by pair and frees one slot before its
//     last pass (eval_mma_slots, eval_slots_main).
// Roles: warp 8 TMA producer, warp 9 MMA issuer (even CTA), warps 0-7
// epilogue (one thread per token and N / 2 columns).
#include <climits>

#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

template <int kM>
struct EvalSmem {
  static constexpr int kN = eval_tile_cols(kM);
  static constexpr int kStages = eval_stages(kM);
  static constexpr uint32_t kBBytes = eval_b_bytes(kM);
  static constexpr uint32_t kA = 0;
  static constexpr uint32_t kB = kStages * kEvalABytes;
  static constexpr uint32_t kX = kA;  // half-merge exchange, after the main loop only
  static constexpr uint32_t kBar = kB + kStages * kBBytes;
  static __device__ __forceinline__ uint32_t full(uint32_t b, int s) { return b + kBar + 8u * s; }
  static __device__ __forceinline__ uint32_t empty(uint32_t b, int s) {
    return b + kBar + 8u * (kStages + s);
  }
  // eight barriers for the accumulators, used as below by each schedule
  static __device__ __forceinline__ uint32_t tb(uint32_t b, int i) {
    return b + kBar + 8u * (2 * kStages + i);
  }
  // all-resident schedule (M != 3): tile j's accumulators are complete: accf(j & 1);
  // the widest sub-model's columns (free0) / all other columns (free1) were read
  static __device__ __forceinline__ uint32_t accf(uint32_t b, int j) { return tb(b, j & 1); }
  static __device__ __forceinline__ uint32_t free0(uint32_t b) { return tb(b, 2); }
  static __device__ __forceinline__ uint32_t free1(uint32_t b) { return tb(b, 3); }
  // slot schedule (M = 3): unit q of the tile is complete (q = 0, 1, 2); unit 0
  // was copied out (copied); the first (pass_a) and second (pass_b) epilogue
  // passes over the last unit are done
  static __device__ __forceinline__ uint32_t unit_full(uint32_t b, int q) { return tb(b, q); }
  static __device__ __forceinline__ uint32_t copied(uint32_t b) { return tb(b, 3); }
  static __device__ __forceinline__ uint32_t pass_a(uint32_t b) { return tb(b, 4); }
  static __device__ __forceinline__ uint32_t pass_b(uint32_t b) { return tb(b, 5); }
  static __device__ __forceinline__ uint32_t drain(uint32_t b) { return tb(b, 7); }
  static constexpr uint32_t kTmemSlot = kBar + 8u * (2 * kStages + 8);
  static constexpr uint32_t kAbort = kTmemSlot + 4;
  static constexpr uint32_t kEnd = kAbort + 4;
  static_assert(kEnd + 1024 <= eval_smem(kM), "eval shared memory map overflows");
  static_assert(eval_slotted(kM) ? 2 * kN <= 512 : kM * kN <= 512,
                "the resident tiles must fit in TMEM");
  static_assert(kBBytes % 1024 == 0, "B stages must stay 1024-byte aligned");
  static_assert((kN / 2) % 16 == 0, "an epilogue thread reads 16-column chunks");
};

constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kDrainNs = 100000000ull;
constexpr int kD = 12;  // field offset of D_sj

// field index of D_sj (j != s) in the partial state
__host__ __device__ constexpr int dfield(int s, int j) { return kD + s * 3 + (j < s ? j : j - 1); }

template <bool kTF32, int kM>
__device__ __forceinline__ void eval_producer(const EvalParams& p, uint32_t base, int row0,
                                              uint32_t rank, int split, volatile int* abort_flag) {
  using Sm = EvalSmem<kM>;
  constexpr int KE = kTF32 ? 32 : 64;
  int stage = 0;
  uint32_t phase = 0, filled = 0, lastpar = 0;
  bool ok = true;
  for (int vt = split; ok && vt < p.nvt; vt += p.S) {
    for (int i = 0; ok && i < kM; ++i) {
      const int m = p.order[i];
      for (int kb = 0; kb < p.nk[m]; ++kb) {
        if (!mbar_wait(Sm::empty(base, stage), phase ^ 1u, abort_flag, p.status)) {
          ok = false;
          break;
        }
        if (rank == 0) mbar_arrive_expect_tx(Sm::full(base, stage), 2 * (kEvalABytes + Sm::kBBytes));
        const uint32_t fb = map_to_rank(Sm::full(base, stage), 0);
        tma_load_2d_pair(base + Sm::kA + stage * kEvalABytes, &p.mapH[m], fb, kb * KE, row0);
        tma_load_2d_pair(base + Sm::kB + stage * Sm::kBBytes, &p.mapW[m], fb, kb * KE,
                         vt * Sm::kN + static_cast<int>(rank) * (Sm::kN / 2));
        filled |= 1u << stage;
        lastpar = (lastpar & ~(1u << stage)) | (phase << stage);
        if (++stage == Sm::kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
  }
  if (!ok && filled) {
    if (rank == 0) {
      for (int s = 0; s < Sm::kStages; ++s)
        if ((filled >> s) & 1u) mbar_wait_drain(Sm::full(base, s), (lastpar >> s) & 1u, kDrainNs, p.status);
    } else {
      spin_ns(kDrainNs);
    }
  }
}

// Unit q of tile j goes to TMEM columns [q N, (q + 1) N).  The widest unit
// (q = 0) of tile j waits for the epilogue to have copied tile j - 1's columns
// of q = 0 (free0); the others wait for it to have finished tile j - 1 (free1).
template <bool kTF32, int kM>
__device__ __forceinline__ void eval_mma(const EvalParams& p, uint32_t base, uint32_t tmem,
                                         int split, volatile int* abort_flag) {
  using Sm = EvalSmem<kM>;
  constexpr uint32_t kIdesc = make_idesc(2 * kHeadBM, Sm::kN, kTF32, false, false);
  int stage = 0;
  uint32_t phase = 0;
  bool ok = true;
  int j = 0;
  for (int vt = split; ok && vt < p.nvt; vt += p.S, ++j) {
    for (int i = 0; ok && i < kM; ++i) {
      const int m = p.order[i];
      if (j > 0 && i <= 1 &&
          !mbar_wait(i == 0 ? Sm::free0(base) : Sm::free1(base), static_cast<uint32_t>(j - 1) & 1u,
                     abort_flag, p.status)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d = tmem + static_cast<uint32_t>(i * Sm::kN);
      for (int kb = 0; kb < p.nk[m]; ++kb) {
        if (!mbar_wait(Sm::full(base, stage), phase, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = make_sdesc(base + Sm::kA + stage * kEvalABytes, 16);
        const uint64_t bd = make_sdesc(base + Sm::kB + stage * Sm::kBBytes, 16);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_issue_pair<kTF32>(d, ad + 2u * kk, bd + 2u * kk, kIdesc, (kb | kk) != 0);
        mma_commit_pair(Sm::empty(base, stage), 0x3);
        if (++stage == Sm::kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    if (!ok) break;
    mma_commit_pair(Sm::accf(base, j), 0x3);
  }
  mma_commit_pair(Sm::drain(base), 0x1);
  mbar_wait_drain(Sm::drain(base), 0, kDrainNs, p.status);
}

// Slot schedule (M = 3).  Tile j's units go to two 256-column TMEM slots,
// a_j = (j & 1) * 256 and b_j = 256 - a_j:
//   unit 0 (widest) -> a_j, after the epilogue's first pass over tile j - 1's
//                      last unit has freed a_j (= b_{j-1})         [pass_a]
//   unit 1 (narrowest) -> b_j, after its second pass has freed b_j   [pass_b]
//   unit 2          -> a_j, once unit 0 has been copied to registers [copied]
// so unit 0 of the next tile, the longest, runs under the end of the epilogue,
// and the pass over units 0 and 1 under unit 2's MMAs.
template <bool kTF32>
__device__ __forceinline__ void eval_mma_slots(const EvalParams& p, uint32_t base, uint32_t tmem,
                                               int split, volatile int* abort_flag) {
  using Sm = EvalSmem<3>;
  constexpr uint32_t kIdesc = make_idesc(2 * kHeadBM, Sm::kN, kTF32, false, false);
  int stage = 0;
  uint32_t phase = 0;
  bool ok = true;
  int j = 0;
  for (int vt = split; ok && vt < p.nvt; vt += p.S, ++j) {
    const uint32_t sa = static_cast<uint32_t>(j & 1) * Sm::kN, sb = Sm::kN - sa;
    for (int i = 0; ok && i < 3; ++i) {
      const int m = p.order[i];
      const uint32_t prev = static_cast<uint32_t>(j - 1) & 1u;
      bool go = true;
      if (i == 0 && j > 0) go = mbar_wait(Sm::pass_a(base), prev, abort_flag, p.status);
      if (i == 1 && j > 0) go = mbar_wait(Sm::pass_b(base), prev, abort_flag, p.status);
      if (i == 2) go = mbar_wait(Sm::copied(base), static_cast<uint32_t>(j) & 1u, abort_flag, p.status);
      if (!go) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d = tmem + (i == 1 ? sb : sa);
      for (int kb = 0; kb < p.nk[m]; ++kb) {
        if (!mbar_wait(Sm::full(base, stage), phase, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = make_sdesc(base + Sm::kA + stage * kEvalABytes, 16);
        const uint64_t bd = make_sdesc(base + Sm::kB + stage * Sm::kBBytes, 16);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          mma_issue_pair<kTF32>(d, ad + 2u * kk, bd + 2u * kk, kIdesc, (kb | kk) != 0);
        mma_commit_pair(Sm::empty(base, stage), 0x3);
        if (++stage == Sm::kStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (ok) mma_commit_pair(Sm::unit_full(base, i), 0x3);
    }
  }
  mma_commit_pair(Sm::drain(base), 0x1);
  mbar_wait_drain(Sm::drain(base), 0, kDrainNs, p.status);
}

// Running state of one thread, indexed by unit position q (sub-model order[q]).
template <int kM>
struct EvalState {
  float m[kM], s[kM];
  int am[kM];
  float d[kM][kM];
};

// 16 columns of every unit's tile: z[q][i] = z_{order[q]} at column col0 + i.
template <int kM, bool kMasked>
__device__ __forceinline__ void eval_chunk(const float (&z)[kM][16], int nvalid, long long col0,
                                           float L1, EvalState<kM>& st) {
#pragma unroll
  for (int q = 0; q < kM; ++q) {
    float cmax = -INFINITY;
    int carg = 0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const bool ok = !kMasked || i < nvalid;
      if (ok && z[q][i] > cmax) {
        cmax = z[q][i];
        carg = i;
      }
    }
    if (cmax > st.m[q]) {
      st.am[q] = static_cast<int>(col0 + carg);
      const float f = st.m[q] == -INFINITY ? 0.f : fast_exp2((st.m[q] - cmax) * L1);
      st.s[q] *= f;
#pragma unroll
      for (int r = 0; r < kM; ++r) st.d[q][r] *= f;
      st.m[q] = cmax;
    }
    const float nb = -st.m[q] * L1;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const bool ok = !kMasked || i < nvalid;
      const float e = ok ? fast_exp2(fmaf(z[q][i], L1, nb)) : 0.f;
      st.s[q] += e;
#pragma unroll
      for (int r = 0; r < kM; ++r)
        if (r != q) st.d[q][r] = fmaf(e, z[q][i] - z[r][i], st.d[q][r]);
    }
  }
}

__device__ __forceinline__ float scale_to(float from, float to, float L1) {
  return from == -INFINITY ? 0.f : fast_exp2((from - to) * L1);
}

// Frees TMEM columns for the MMA issuer: every epilogue warp of both CTAs
// arrives on the even CTA's barrier once its reads have completed.
__device__ __forceinline__ void eval_release(uint32_t bar, int lane) {
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive_remote(map_to_rank(bar, 0));
}

// ---- slot schedule epilogue (M = 3)
// Columns past V take this logit: exp2 of it underflows to 0 against any real
// maximum, it never wins a maximum over a chunk that has a valid column, and
// two of them differ by 0, so every accumulation ignores them without a
// second (masked) copy of the code.
constexpr float kPadLogit = -1e30f;

// This thread's 16 columns at TMEM address t; columns from nvalid on padded.
__device__ __forceinline__ void ld_chunk(uint32_t t, int nvalid, float (&z)[16]) {
  tmem_ld16(t, z);
  if (nvalid < 16) {
#pragma unroll
    for (int i = 0; i < 16; ++i)
      if (i >= nvalid) z[i] = kPadLogit;
  }
}
// Two chunks in one wait: na (nb) of a's (b's) columns are valid.
__device__ __forceinline__ void ld_chunk2(uint32_t ta, uint32_t tb, int na, int nb, float (&a)[16],
                                          float (&b)[16]) {
  tmem_ld16x2(ta, tb, a, b);
  if (na < 16 || nb < 16) {
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      if (i >= na) a[i] = kPadLogit;
      if (i >= nb) b[i] = kPadLogit;
    }
  }
}

// Maximum of a chunk and the first column attaining it, by a tree whose left
// operand always holds the lower columns (ties keep the left one).
__device__ __forceinline__ void chunk_argmax(const float (&z)[16], float& vmax, int& imax) {
  float v[8];
  int ix[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const bool r = z[2 * k + 1] > z[2 * k];
    v[k] = r ? z[2 * k + 1] : z[2 * k];
    ix[k] = r ? 2 * k + 1 : 2 * k;
  }
#pragma unroll
  for (int w = 4; w >= 1; w >>= 1) {
#pragma unroll
    for (int k = 0; k < w; ++k) {
      const bool r = v[2 * k + 1] > v[2 * k];
      v[k] = r ? v[2 * k + 1] : v[2 * k];
      ix[k] = r ? ix[2 * k + 1] : ix[2 * k];
    }
  }
  vmax = v[0];
  imax = ix[0];
}

// Folds a tile's maximum (tmax at column tcol) into unit q's running state:
// a new maximum rescales the unit's sum and its D_q*.
__device__ __forceinline__ void fold_max(EvalState<3>& st, int q, float tmax, long long tcol, float L1) {
  if (tmax > st.m[q]) {
    st.am[q] = static_cast<int>(tcol);
    const float f = st.m[q] == -INFINITY ? 0.f : fast_exp2((st.m[q] - tmax) * L1);
    st.s[q] *= f;
#pragma unroll
    for (int r = 0; r < 3; ++r) st.d[q][r] *= f;
    st.m[q] = tmax;
  }
}

// Tile maximum of a unit held in TMEM at t (this thread's 128 columns).
__device__ __forceinline__ void tmem_tile_max(uint32_t t, long long tcol, long long V, float& tmax,
                                              long long& targ) {
  tmax = -INFINITY;
  targ = 0;
#pragma unroll
  for (int c = 0; c < 8; c += 2) {
    const long long col0 = tcol + c * 16;
    if (col0 >= V) continue;  // warp-uniform
    float za[16], zb[16];
    ld_chunk2(t + static_cast<uint32_t>(c * 16), t + static_cast<uint32_t>(c * 16 + 16),
              static_cast<int>(min(16LL, V - col0)), static_cast<int>(max(0LL, min(16LL, V - col0 - 16))),
              za, zb);
    float va, vb;
    int ia, ib;
    chunk_argmax(za, va, ia);
    chunk_argmax(zb, vb, ib);
    if (col0 + 16 >= V) vb = -INFINITY;  // the second chunk is past V
    if (va > tmax) {
      tmax = va;
      targ = col0 + ia;
    }
    if (vb > tmax) {
      tmax = vb;
      targ = col0 + 16 + ib;
    }
  }
}

// Partial sums of one pass over one pair (a, b) with both maxima fixed.
struct PairSums {
  float sa0, sa1, sb0, sb1, dab0, dab1, dba0, dba1;
};

// One 16-column chunk of pair (a, b): e_a, e_b against the fixed maxima
// (na = -m_a log2 e, nb = -m_b log2 e); two interleaved partials per sum.
template <bool kSumA, bool kSumB>
__device__ __forceinline__ void pair_chunk(const float (&za)[16], const float (&zb)[16], float L1,
                                           float na, float nb, PairSums& ps) {
#pragma unroll
  for (int i = 0; i < 16; i += 2) {
    const float ea0 = fast_exp2(fmaf(za[i], L1, na)), ea1 = fast_exp2(fmaf(za[i + 1], L1, na));
    const float eb0 = fast_exp2(fmaf(zb[i], L1, nb)), eb1 = fast_exp2(fmaf(zb[i + 1], L1, nb));
    const float d0 = za[i] - zb[i], d1 = za[i + 1] - zb[i + 1];
    if (kSumA) {
      ps.sa0 += ea0;
      ps.sa1 += ea1;
    }
    if (kSumB) {
      ps.sb0 += eb0;
      ps.sb1 += eb1;
    }
    ps.dab0 = fmaf(ea0, d0, ps.dab0);
    ps.dab1 = fmaf(ea1, d1, ps.dab1);
    ps.dba0 = fmaf(eb0, -d0, ps.dba0);
    ps.dba1 = fmaf(eb1, -d1, ps.dba1);
  }
}

template <bool kSumA, bool kSumB>
__device__ __forceinline__ void fold_pair(EvalState<3>& st, int a, int b, const PairSums& ps) {
  if (kSumA) st.s[a] += ps.sa0 + ps.sa1;
  if (kSumB) st.s[b] += ps.sb0 + ps.sb1;
  st.d[a][b] += ps.dab0 + ps.dab1;
  st.d[b][a] += ps.dba0 + ps.dba1;
}

// Per tile (slots as in eval_mma_slots):
//   copy    unit 0 into registers (padded past V), its tile maximum; release (copied)
//   pass 1  (units 0, 1)  unit 1's tile maximum, then the sums of both, D_01, D_10
//           [under unit 2's MMAs]
//   pass 2a (units 1, 2)  unit 2's tile maximum, then its sum, D_12, D_21; release b_j
//   pass 2b (units 0, 2)  D_02, D_20; release a_j    [under the next tile's unit 0]
// Every pass runs with its units' maxima already folded in, so its chunks are
// independent of one another.
__device__ __forceinline__ bool eval_slots_main(const EvalParams& p, uint32_t base, uint32_t tl,
                                                int split, int half, int lane,
                                                volatile int* abort_flag, EvalState<3>& st) {
  using Sm = EvalSmem<3>;
  constexpr int kHalf = Sm::kN / 2;  // 128 columns per thread
  constexpr int kChunks = kHalf / 16;
  const float L1 = p.L1;
  const long long V = p.V;
  int j = 0;
  for (int vt = split; vt < p.nvt; vt += p.S, ++j) {
    const uint32_t par = static_cast<uint32_t>(j) & 1u;
    const uint32_t sa = par * Sm::kN, sb = Sm::kN - sa;
    const long long tcol = static_cast<long long>(vt) * Sm::kN + half * kHalf;
    bool ok = mbar_wait(Sm::unit_full(base, 0), par, abort_flag, p.status);
    if (!__all_sync(0xffffffffu, ok)) return false;
    tc_fence_after();
    float z0[kChunks][16];
#pragma unroll
    for (int c = 0; c < kChunks; c += 2)
      tmem_ld16x2(tl + sa + static_cast<uint32_t>(c * 16), tl + sa + static_cast<uint32_t>(c * 16 + 16),
                  z0[c], z0[c + 1]);
    eval_release(Sm::copied(base), lane);
    {
      float tmax = -INFINITY;
      long long targ = 0;
#pragma unroll
      for (int c = 0; c < kChunks; ++c) {
        const long long col0 = tcol + c * 16;
        if (col0 + 16 > V) {
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (col0 + i >= V) z0[c][i] = kPadLogit;
        }
        if (col0 >= V) continue;
        float v;
        int ix;
        chunk_argmax(z0[c], v, ix);
        if (v > tmax) {
          tmax = v;
          targ = col0 + ix;
        }
      }
      fold_max(st, 0, tmax, targ, L1);
    }

    ok = mbar_wait(Sm::unit_full(base, 1), par, abort_flag, p.status);
    if (!__all_sync(0xffffffffu, ok)) return false;
    tc_fence_after();
    {
      float tmax;
      long long targ;
      tmem_tile_max(tl + sb, tcol, V, tmax, targ);
      fold_max(st, 1, tmax, targ, L1);
      const float n0 = -st.m[0] * L1, n1 = -st.m[1] * L1;
      PairSums ps = {};
#pragma unroll
      for (int c = 0; c < kChunks; ++c) {
        const long long col0 = tcol + c * 16;
        if (col0 >= V) continue;  // warp-uniform
        float z1[16];
        ld_chunk(tl + sb + static_cast<uint32_t>(c * 16), static_cast<int>(min(16LL, V - col0)), z1);
        pair_chunk<true, true>(z0[c], z1, L1, n0, n1, ps);
      }
      fold_pair<true, true>(st, 0, 1, ps);
    }

    ok = mbar_wait(Sm::unit_full(base, 2), par, abort_flag, p.status);
    if (!__all_sync(0xffffffffu, ok)) return false;
    tc_fence_after();
    {
      float tmax;
      long long targ;
      tmem_tile_max(tl + sa, tcol, V, tmax, targ);
      fold_max(st, 2, tmax, targ, L1);
      const float n1 = -st.m[1] * L1, n2 = -st.m[2] * L1;
      PairSums ps = {};
#pragma unroll
      for (int c = 0; c < kChunks; ++c) {
        const long long col0 = tcol + c * 16;
        if (col0 >= V) continue;
        float z1[16], z2[16];
        const int nv = static_cast<int>(min(16LL, V - col0));
        ld_chunk2(tl + sb + static_cast<uint32_t>(c * 16), tl + sa + static_cast<uint32_t>(c * 16), nv, nv,
                  z1, z2);
        pair_chunk<false, true>(z1, z2, L1, n1, n2, ps);
      }
      fold_pair<false, true>(st, 1, 2, ps);
    }
    eval_release(Sm::pass_a(base), lane);
    {
      const float n0 = -st.m[0] * L1, n2 = -st.m[2] * L1;
      PairSums ps = {};
#pragma unroll
      for (int c = 0; c < kChunks; ++c) {
        const long long col0 = tcol + c * 16;
        if (col0 >= V) continue;
        float z2[16];
        ld_chunk(tl + sa + static_cast<uint32_t>(c * 16), static_cast<int>(min(16LL, V - col0)), z2);
        pair_chunk<false, false>(z0[c], z2, L1, n0, n2, ps);
      }
      fold_pair<false, false>(st, 0, 2, ps);
    }
    eval_release(Sm::pass_b(base), lane);
  }
  return true;
}

template <int kM>
__device__ __forceinline__ void eval_epilogue(const EvalParams& p, uint32_t base, uint32_t tmem,
                                              float* xchg, int row_base, int split, int warp,
                                              int lane, volatile int* abort_flag) {
  using Sm = EvalSmem<kM>;
  constexpr int kHalf = Sm::kN / 2;  // columns per thread
  constexpr int kChunks = kHalf / 16;
  const int quad = warp & 3, half = warp >> 2;
  const int r = quad * 32 + lane;
  const long long row = static_cast<long long>(row_base) + r;
  const uint32_t tl = tmem + (static_cast<uint32_t>(quad * 32) << 16) + static_cast<uint32_t>(half * kHalf);
  const float L1 = p.L1;
  EvalState<kM> st;
#pragma unroll
  for (int q = 0; q < kM; ++q) {
    st.m[q] = -INFINITY;
    st.s[q] = 0.f;
    st.am[q] = 0;
#pragma unroll
    for (int j = 0; j < kM; ++j) st.d[q][j] = 0.f;
  }
  if constexpr (eval_slotted(kM)) {
    eval_slots_main(p, base, tl, split, half, lane, abort_flag, st);
  } else {
  int j = 0;
  for (int vt = split; vt < p.nvt; vt += p.S, ++j) {
    const bool ok = mbar_wait(Sm::accf(base, j), static_cast<uint32_t>(j >> 1) & 1u, abort_flag, p.status);
    if (!__all_sync(0xffffffffu, ok)) break;
    tc_fence_after();
    // the widest unit's columns into registers, then its TMEM columns are free
    float z0[kChunks][16];
#pragma unroll
    for (int c = 0; c < kChunks; ++c) tmem_ld16(tl + static_cast<uint32_t>(c * 16), z0[c]);
    eval_release(Sm::free0(base), lane);
#pragma unroll
    for (int c = 0; c < kChunks; ++c) {
      const long long col0 = static_cast<long long>(vt) * Sm::kN + half * kHalf + c * 16;
      const int nvalid = static_cast<int>(max(0LL, min(16LL, p.V - col0)));
      if (nvalid == 0) continue;  // warp-uniform
      float z[kM][16];
#pragma unroll
      for (int i = 0; i < 16; ++i) z[0][i] = z0[c][i];
#pragma unroll
      for (int q = 1; q < kM; ++q) tmem_ld16(tl + static_cast<uint32_t>(q * Sm::kN + c * 16), z[q]);
      if (nvalid == 16)
        eval_chunk<kM, false>(z, 16, col0, L1, st);
      else
        eval_chunk<kM, true>(z, nvalid, col0, L1, st);
    }
    eval_release(Sm::free1(base), lane);
  }
  }

  // The two column halves of a token combine through shared memory; fields
  // are indexed by sub-model (order[q]).
  auto X = [&](int f) -> float& { return xchg[f * kHeadBM + r]; };
  if (half == 1) {
#pragma unroll
    for (int q = 0; q < kM; ++q) {
      const int s = p.order[q];
      X(s) = st.m[q];
      X(4 + s) = st.s[q];
      X(8 + s) = __int_as_float(st.am[q]);
#pragma unroll
      for (int q2 = 0; q2 < kM; ++q2)
        if (q2 != q) X(dfield(s, p.order[q2])) = st.d[q][q2];
    }
  }
  named_bar_sync(1, kHeadEpiWarps * 32);
  if (half == 1 || row >= p.T) return;
  float* P = p.part + static_cast<long long>(split) * kEvalFields * p.T + row;
#pragma unroll
  for (int q = 0; q < kM; ++q) {
    const int s = p.order[q];
    const float m1 = X(s), mm = fmaxf(st.m[q], m1);
    const float fa = scale_to(st.m[q], mm, L1), fb = scale_to(m1, mm, L1);
    const int a1 = __float_as_int(X(8 + s));
    P[s * p.T] = mm;
    P[(4 + s) * p.T] = st.s[q] * fa + X(4 + s) * fb;
    P[(8 + s) * p.T] = __int_as_float(m1 > st.m[q] ? a1 : (st.m[q] > m1 ? st.am[q] : min(st.am[q], a1)));
#pragma unroll
    for (int q2 = 0; q2 < kM; ++q2)
      if (q2 != q) {
        const int f = dfield(s, p.order[q2]);
        P[f * p.T] = st.d[q][q2] * fa + X(f) * fb;
      }
  }
}

template <bool kTF32, int kM>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kHeadThreads, 1)
    eval_kernel(const __grid_constant__ EvalParams p) {
  using Sm = EvalSmem<kM>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(gbase + Sm::kAbort);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + Sm::kTmemSlot);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  int tt, split;
  band_unit(static_cast<int>(blockIdx.x >> 1), p.ntt, p.S, p.band, tt, split);
  const int row_base = tt * 2 * kHeadBM + static_cast<int>(rank) * kHeadBM;

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int s = 0; s < Sm::kStages; ++s) {
      mbar_init(Sm::full(base, s), 1);
      mbar_init(Sm::empty(base, s), 1);
    }
    if constexpr (eval_slotted(kM)) {
      for (int q = 0; q < 3; ++q) mbar_init(Sm::unit_full(base, q), 1);
      mbar_init(Sm::copied(base), 2 * kHeadEpiWarps);
      mbar_init(Sm::pass_a(base), 2 * kHeadEpiWarps);
      mbar_init(Sm::pass_b(base), 2 * kHeadEpiWarps);
    } else {
      for (int q = 0; q < 2; ++q) mbar_init(Sm::accf(base, q), 1);
      mbar_init(Sm::free0(base), 2 * kHeadEpiWarps);
      mbar_init(Sm::free1(base), 2 * kHeadEpiWarps);
    }
    mbar_init(Sm::drain(base), 1);
    fence_barrier_init();
  }
  if (warp == kHeadEpiWarps + 1) {
    tmem_alloc_pair(base + Sm::kTmemSlot, kTmemCols);
    tmem_relinquish_pair();
  }
  if (warp == kHeadEpiWarps && lane == 0) {
    for (int m = 0; m < kM; ++m) {
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
      if (lane == 0) eval_producer<kTF32, kM>(p, base, row_base, rank, split, abort_flag);
    } else if (warp == kHeadEpiWarps + 1) {
      if (lane == 0 && rank == 0) {
        if constexpr (eval_slotted(kM))
          eval_mma_slots<kTF32>(p, base, tmem, split, abort_flag);
        else
          eval_mma<kTF32, kM>(p, base, tmem, split, abort_flag);
      }
      __syncwarp();
    }
  } else {
    regs_increase<kHeadEpiRegs>();
    eval_epilogue<kM>(p, base, tmem, reinterpret_cast<float*>(gbase + Sm::kX), row_base, split,
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

template <int kM>
cudaError_t launch_eval_m(const EvalParams& p, bool tf32, int grid, cudaStream_t s) {
  if (tf32)
    eval_kernel<true, kM><<<grid, kHeadThreads, eval_smem(kM), s>>>(p);
  else
    eval_kernel<false, kM><<<grid, kHeadThreads, eval_smem(kM), s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_eval(const EvalParams& p, bool tf32, cudaStream_t s) {
  const int grid = 2 * p.ntt * p.S;
  if (grid <= 0) return cudaSuccess;
  switch (p.M) {
    case 1: return launch_eval_m<1>(p, tf32, grid, s);
    case 2: return launch_eval_m<2>(p, tf32, grid, s);
    case 3: return launch_eval_m<3>(p, tf32, grid, s);
    default: return launch_eval_m<4>(p, tf32, grid, s);
  }
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
#define MLS_SET(TF, M)                                                                        \
  e = cudaFuncSetAttribute(eval_kernel<TF, M>, cudaFuncAttributeMaxDynamicSharedMemorySize,   \
                           eval_smem(M));                                                     \
  if (e != cudaSuccess) return e;                                                             \
  {                                                                                           \
    cudaFuncAttributes fa;                                                                    \
    e = cudaFuncGetAttributes(&fa, eval_kernel<TF, M>);                                       \
    if (e != cudaSuccess) return e;                                                           \
    if (fa.maxThreadsPerBlock < kHeadThreads || fa.numRegs != kHeadLaunchRegs)                \
      return cudaErrorLaunchOutOfResources;                                                   \
  }
  MLS_SET(true, 1)
  MLS_SET(true, 2)
  MLS_SET(true, 3)
  MLS_SET(true, 4)
  MLS_SET(false, 1)
  MLS_SET(false, 2)
  MLS_SET(false, 3)
  MLS_SET(false, 4)
#undef MLS_SET
  return cudaSuccess;
}

}  // namespace mls
