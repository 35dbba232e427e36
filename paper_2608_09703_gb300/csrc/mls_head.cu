// Fused LM-head kernels of the Matryoshka-suite output stage.
//
// A CTA pair (cluster of 2) owns 256 tokens and a strided set of 256-column
// vocabulary tiles.  For every vocabulary tile it computes the teacher's logit
// tile z_t = H_t W_t^T first and then each student's z_m = H_m W_m^T (Sec. 2:
// each sub-model has its own head W^m in R^{V x D_m}), on the tensor cores:
//
//   warp 8   TMA producer (each CTA): its 128 token rows of H_m and its 128
//            vocabulary rows of W_m, k-blocks of 128 bytes, into a 6-stage
//            128B-swizzled ring; both CTAs' loads complete on the even CTA's
//            barrier
//   warp 9   MMA issuer (even CTA): pair tcgen05.mma 256x256xK (cta_group::2)
//            into one of two TMEM accumulators (2 x 256 columns in each CTA),
//            commits multicast to both CTAs
//   warps 0-7 epilogue: tcgen05.ld, one thread per (token, half tile); these
//            two warpgroups take the registers the third one gives up, since
//            each thread keeps the teacher's 128 weights of a tile in registers
//
// The epilogue never writes a logit to memory:
//   forward  (Eq. 2 and Eq. 3): single-pass online logsumexp of z (tau = 1)
//            and of z / tau, the teacher weights q~ = exp((z_t - max_t)/tau)
//            kept in registers for the tile, the teacher-weighted sums
//            A_m = sum_v q~_v z_m[v] (rescaled when the teacher's running max
//            moves), the target logit and a running argmax.  The two threads
//            of a token (one per column half) combine their states through
//            shared memory and each CTA writes one partial state per
//            (token, model); a merge kernel combines the CTAs' partials.
//   backward recomputes the same tiles and forms dL/dz in registers:
//            teacher  c_t (softmax(z_t) - e_y)                (stop-grad on q)
//            student  c_m [(1-alpha)(softmax(z_m) - e_y) + (alpha/tau)(softmax(z_m/tau) - q)]
//            with q = softmax(z_t / tau) from the forward's statistics, and
//            stores it (bf16, fp32 for fp32 inputs) for the dH / dW GEMMs.
#include "mls_device.cuh"
#include "mls_kernels.h"

namespace mls {
namespace {

constexpr int kModeFwd = 0;
constexpr int kModeBwd = 1;
constexpr int kStud = kMaxModels - 1;

// Shared-memory map, offsets from the 1024-byte-aligned base.
struct HeadSmem {
  static constexpr uint32_t kA = 0;
  static constexpr uint32_t kB = kHeadStages * kHeadABytes;
  static constexpr uint32_t kStage = kB + kHeadStages * kHeadBBytes;  // dL/dz staging
  static constexpr uint32_t kBar = kStage + kHeadStaging;
  static __device__ __forceinline__ uint32_t full(uint32_t b, int s) { return b + kBar + 8u * s; }
  static __device__ __forceinline__ uint32_t empty(uint32_t b, int s) {
    return b + kBar + 8u * (kHeadStages + s);
  }
  static __device__ __forceinline__ uint32_t accf(uint32_t b, uint32_t a) {
    return b + kBar + 8u * (2 * kHeadStages + a);
  }
  static __device__ __forceinline__ uint32_t acce(uint32_t b, uint32_t a) {
    return b + kBar + 8u * (2 * kHeadStages + 2 + a);
  }
  static __device__ __forceinline__ uint32_t drain(uint32_t b) {
    return b + kBar + 8u * (2 * kHeadStages + 4);
  }
  static constexpr uint32_t kTmemSlot = kBar + 8u * (2 * kHeadStages + 5);
  static constexpr uint32_t kAbort = kTmemSlot + 4;
  static constexpr uint32_t kEnd = kAbort + 4;
};
static_assert(HeadSmem::kEnd + 1024 <= kHeadSmem, "head shared memory map overflows");
static_assert(kPartFields * kMaxModels * kHeadBM * 4 <= kHeadStaging,
              "forward half-merge exchange must fit in the staging area");

constexpr uint32_t kTmemCols = 512;             // two 256-column fp32 accumulators
constexpr uint64_t kDrainNs = 100000000ull;     // bound for shutdown waits

// ------------------------------------------------------------------ producer
template <bool kTF32>
__device__ __forceinline__ void head_producer(const HeadParams& p, uint32_t base, int row0,
                                              uint32_t rank, int split, volatile int* abort_flag) {
  constexpr int KE = kTF32 ? 32 : 64;  // elements in 128 bytes of K
  int stage = 0;
  uint32_t phase = 0, filled = 0, lastpar = 0;
  bool ok = true;
  // Test hook (off unless the host sets it): the first pair issues nothing for
  // its first stage, so the MMA issuer's wait on that stage must run out.
  bool stall = p.test_stall && (blockIdx.x >> 1) == 0;
  for (int vt = p.vt_begin + split; ok && vt < p.vt_end; vt += p.S) {
    for (int u = 0; ok && u < p.M; ++u) {
      const int m = p.order[u];
      MLS_CHECK(p.status, m >= 0 && m < p.M && split < p.S &&
                              static_cast<long long>(vt) * kHeadBN < p.V + kHeadBN);
      for (int kb = 0; kb < p.nk[m]; ++kb) {
        if (!mbar_wait(HeadSmem::empty(base, stage), phase ^ 1u, abort_flag, p.status)) {
          ok = false;
          break;
        }
        if (stall) {
          stall = false;
          if (++stage == kHeadStages) {
            stage = 0;
            phase ^= 1u;
          }
          continue;
        }
        // both CTAs' halves are counted on the even CTA's barrier
        if (rank == 0) mbar_arrive_expect_tx(HeadSmem::full(base, stage), 2 * (kHeadABytes + kHeadBBytes));
        const uint32_t fb = map_to_rank(HeadSmem::full(base, stage), 0);
        tma_load_2d_pair(base + HeadSmem::kA + stage * kHeadABytes, &p.mapH[m], fb, kb * KE, row0);
        tma_load_2d_pair(base + HeadSmem::kB + stage * kHeadBBytes, &p.mapW[m], fb, kb * KE,
                         vt * kHeadBN + static_cast<int>(rank) * kHeadBHalf);
        filled |= 1u << stage;
        lastpar = (lastpar & ~(1u << stage)) | (phase << stage);
        if (++stage == kHeadStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
  }
  if (!ok && filled) {
    // Loads already issued must land before this CTA's shared memory goes away.
    // The even CTA can watch its barriers; the odd CTA's loads are counted on
    // the even CTA's barriers, so it waits out a bound no TMA load approaches.
    if (rank == 0) {
      for (int s = 0; s < kHeadStages; ++s)
        if ((filled >> s) & 1u) mbar_wait_drain(HeadSmem::full(base, s), (lastpar >> s) & 1u, kDrainNs, p.status);
    } else {
      spin_ns(kDrainNs);
    }
  }
}

// ------------------------------------------------------------------ MMA issuer
template <bool kTF32>
__device__ __forceinline__ void head_mma(const HeadParams& p, uint32_t base, uint32_t tmem,
                                         int split, volatile int* abort_flag) {
  constexpr uint32_t kIdesc = make_idesc(2 * kHeadBM, kHeadBN, kTF32, false, false);
  constexpr uint16_t kBoth = 0x3;
  int stage = 0;
  uint32_t phase = 0, acc = 0, acc_par = 0;
  bool ok = true;
  for (int vt = p.vt_begin + split; ok && vt < p.vt_end; vt += p.S) {
    for (int u = 0; ok && u < p.M; ++u) {
      const int m = p.order[u];
      if (!mbar_wait(HeadSmem::acce(base, acc), acc_par ^ 1u, abort_flag, p.status)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t d = tmem + acc * kHeadBN;
      for (int kb = 0; kb < p.nk[m]; ++kb) {
        if (!mbar_wait(HeadSmem::full(base, stage), phase, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t ad = make_sdesc(base + HeadSmem::kA + stage * kHeadABytes, 16);
        const uint64_t bd = make_sdesc(base + HeadSmem::kB + stage * kHeadBBytes, 16);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)  // 4 x 32 bytes of K per stage
          mma_issue_pair<kTF32>(d, ad + 2u * kk, bd + 2u * kk, kIdesc, (kb | kk) != 0);
        mma_commit_pair(HeadSmem::empty(base, stage), kBoth);
        if (++stage == kHeadStages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      if (!ok) break;
      mma_commit_pair(HeadSmem::accf(base, acc), kBoth);
      acc ^= 1u;
      if (acc == 0) acc_par ^= 1u;
    }
  }
  // Every MMA this thread issued has finished before TMEM is released.
  mma_commit_pair(HeadSmem::drain(base), 0x1);
  mbar_wait_drain(HeadSmem::drain(base), 0, kDrainNs, p.status);
}

// Waits for accumulator `acc` to be full; warp-uniform result.
__device__ __forceinline__ bool epi_acquire(const HeadParams& p, uint32_t base, uint32_t acc,
                                            uint32_t acc_par, volatile int* abort_flag) {
  const bool ok = mbar_wait(HeadSmem::accf(base, acc), acc_par, abort_flag, p.status);
  const bool all = __all_sync(0xffffffffu, ok);
  tc_fence_after();
  return all;
}

__device__ __forceinline__ void epi_release(uint32_t base, uint32_t& acc, uint32_t& acc_par,
                                            int lane) {
  tc_fence_before();
  __syncwarp();
  if (lane == 0) mbar_arrive_remote(map_to_rank(HeadSmem::acce(base, acc), 0));
  acc ^= 1u;
  if (acc == 0) acc_par ^= 1u;
}

// ------------------------------------------------------------------ forward epilogue
// Teacher tile: two passes over the thread's 128 columns.  Pass 1 finds the
// tile maximum (and argmax); the running statistics and every student's
// teacher-weighted sum are rescaled to the new maximum; pass 2 accumulates
// the exponentials and leaves q~_v = exp((z_t[v] - max_t) / tau) in q[].
// The teacher's own weighted sum is kept relative to its running maximum,
// acc = sum_v q~_v (z_t[v] - max_t) log2(e) / tau (every term <= 0), so that the
// entropy H(q) = log S - acc / (S log2(e)) is formed without cancellation even
// when q is sharply peaked.
template <bool kMasked, bool kTauOne>
__device__ __forceinline__ void fwd_teacher(uint32_t ta, int nvalid, int yl, long long col0,
                                            float L1, float Lt, float& m, float& s1, float& st,
                                            float& acc, float& zy, int& am, float (&q)[128],
                                            float (&aS)[kStud]) {
  float v[32];
  float tmax = -INFINITY;
  int targ = 0;
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    if (kMasked && c * 32 >= nvalid) break;
    tmem_ld32(ta + c * 32, v);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const bool ok = !kMasked || (c * 32 + i < nvalid);
      if (ok && v[i] > tmax) {
        tmax = v[i];
        targ = c * 32 + i;
      }
    }
  }
  if (tmax > m) am = static_cast<int>(col0 + targ);
  const float mn = fmaxf(m, tmax);
  const float sc1 = fast_exp2((m - mn) * L1);
  const float sct = kTauOne ? sc1 : fast_exp2((m - mn) * Lt);
  const float st_old = kTauOne ? s1 : st;
  if (st_old > 0.f) acc = sct * (acc + (m - mn) * Lt * st_old);
  s1 *= sc1;
  if (!kTauOne) st *= sct;
#pragma unroll
  for (int j = 0; j < kStud; ++j) aS[j] *= sct;
  m = mn;
  const float b1 = -mn * L1, bt = -mn * Lt;
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    if (kMasked && c * 32 >= nvalid) {
#pragma unroll
      for (int i = 0; i < 32; ++i) q[c * 32 + i] = 0.f;
      continue;
    }
    tmem_ld32(ta + c * 32, v);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const bool ok = !kMasked || (c * 32 + i < nvalid);
      const float z = ok ? v[i] : -INFINITY;
      const float x1 = fmaf(z, L1, b1);
      const float xt = kTauOne ? x1 : fmaf(z, Lt, bt);
      const float e1 = fast_exp2(x1);
      const float et = kTauOne ? e1 : fast_exp2(xt);
      s1 += e1;
      if (!kTauOne) st += et;
      acc = fmaf(et, ok ? xt : 0.f, acc);
      q[c * 32 + i] = et;
    }
    const int r = yl - c * 32;
    if (static_cast<unsigned>(r) < 32u) {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (i == r) zy = v[i];
    }
  }
}

// Student tile: one pass, online per 32-column chunk.  Its teacher-weighted
// sum uses the q~ of the same vocabulary tile, relative to the teacher's
// current running maximum.
template <bool kMasked, bool kTauOne>
__device__ __forceinline__ void fwd_student(uint32_t ta, int nvalid, int yl, long long col0,
                                            float L1, float Lt, float& m, float& s1, float& st,
                                            float& acc, float& zy, int& am, const float (&q)[128]) {
  float v[32];
#pragma unroll
  for (int c = 0; c < 4; ++c) {
    if (kMasked && c * 32 >= nvalid) break;
    tmem_ld32(ta + c * 32, v);
    float cmax = -INFINITY;
    int carg = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const bool ok = !kMasked || (c * 32 + i < nvalid);
      if (ok && v[i] > cmax) {
        cmax = v[i];
        carg = i;
      }
    }
    if (cmax > m) {
      am = static_cast<int>(col0 + c * 32 + carg);
      s1 *= fast_exp2((m - cmax) * L1);
      if (!kTauOne) st *= fast_exp2((m - cmax) * Lt);
      m = cmax;
    }
    const float b1 = -m * L1, bt = -m * Lt;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const bool ok = !kMasked || (c * 32 + i < nvalid);
      const float z = ok ? v[i] : -INFINITY;
      s1 += fast_exp2(fmaf(z, L1, b1));
      if (!kTauOne) st += fast_exp2(fmaf(z, Lt, bt));
      acc = fmaf(q[c * 32 + i], ok ? v[i] : 0.f, acc);
    }
    const int r = yl - c * 32;
    if (static_cast<unsigned>(r) < 32u) {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (i == r) zy = v[i];
    }
  }
}

// Combines the row state of the other column half (b) into this one (a):
// both are rescaled to the larger running maximum.
struct RowState {
  float m, s1, st, acc, zy;
  int am;
};

__device__ __forceinline__ float scale_from(float from, float to, float L) {
  return from == -INFINITY ? 0.f : fast_exp2((from - to) * L);
}

// Argmax of two halves: the larger maximum, the lower index on a tie.
__device__ __forceinline__ int merged_argmax(float ma, int aa, float mb, int ab) {
  if (mb > ma) return ab;
  if (ma > mb) return aa;
  return aa < ab ? aa : ab;
}

template <bool kTauOne>
__device__ __forceinline__ void fwd_epilogue(const HeadParams& p, uint32_t base, uint32_t tmem,
                                             float* xchg, int row_base, int split, int warp,
                                             int lane, volatile int* abort_flag) {
  const int quad = warp & 3, half = warp >> 2;
  const long long row = static_cast<long long>(row_base) + quad * 32 + lane;
  const bool row_ok = row < p.T;
  const int y = row_ok ? __ldg(p.y + row) : -1;
  const uint32_t tl = tmem + (static_cast<uint32_t>(quad * 32) << 16) + static_cast<uint32_t>(half * 128);
  const float L1 = p.L1, Lt = p.Ltau;
  const int nst = p.M - 1;

  float mT = -INFINITY, s1T = 0.f, stT = 0.f, aT = 0.f, zT = 0.f;
  int amT = 0;
  float mS[kStud], s1S[kStud], stS[kStud], aS[kStud], zS[kStud];
  int amS[kStud];
#pragma unroll
  for (int j = 0; j < kStud; ++j) {
    mS[j] = -INFINITY;
    s1S[j] = stS[j] = aS[j] = zS[j] = 0.f;
    amS[j] = 0;
  }
  float q[128];
  uint32_t acc = 0, acc_par = 0;

  bool aborted = false;
  for (int vt = p.vt_begin + split; !aborted && vt < p.vt_end; vt += p.S) {
    const long long col0 = static_cast<long long>(vt) * kHeadBN + half * 128;
    const int nvalid = static_cast<int>(max(0LL, min(128LL, p.V - col0)));
    const int yl = y >= 0 ? static_cast<int>(y - col0) : -1;

    if (!epi_acquire(p, base, acc, acc_par, abort_flag)) break;
    {
      const uint32_t ta = tl + acc * kHeadBN;
      if (nvalid == 128)
        fwd_teacher<false, kTauOne>(ta, 128, yl, col0, L1, Lt, mT, s1T, stT, aT, zT, amT, q, aS);
      else if (nvalid > 0)
        fwd_teacher<true, kTauOne>(ta, nvalid, yl, col0, L1, Lt, mT, s1T, stT, aT, zT, amT, q, aS);
      else {
#pragma unroll
        for (int i = 0; i < 128; ++i) q[i] = 0.f;
      }
    }
    epi_release(base, acc, acc_par, lane);

#pragma unroll
    for (int j = 0; j < kStud; ++j) {
      if (j < nst && !aborted) {
        if (!epi_acquire(p, base, acc, acc_par, abort_flag)) {
          aborted = true;
          break;
        }
        const uint32_t ta = tl + acc * kHeadBN;
        if (nvalid == 128)
          fwd_student<false, kTauOne>(ta, 128, yl, col0, L1, Lt, mS[j], s1S[j], stS[j], aS[j],
                                      zS[j], amS[j], q);
        else if (nvalid > 0)
          fwd_student<true, kTauOne>(ta, nvalid, yl, col0, L1, Lt, mS[j], s1S[j], stS[j], aS[j],
                                     zS[j], amS[j], q);
        epi_release(base, acc, acc_par, lane);
      }
    }
  }
  if (kTauOne) {
    stT = s1T;
#pragma unroll
    for (int j = 0; j < kStud; ++j) stS[j] = s1S[j];
  }

  // The two threads of a token (warps w and w + 4) hold the states of the two
  // column halves; the second hands its state over through shared memory
  // (xchg[field][slot][128 rows]) and the first writes the CTA's partial.
  const int r = quad * 32 + lane;
  auto X = [&](int f, int slot) -> float& { return xchg[(f * kMaxModels + slot) * kHeadBM + r]; };
  if (half == 1) {
    X(kPartMax, 0) = mT; X(kPartSum1, 0) = s1T; X(kPartSumTau, 0) = stT;
    X(kPartAcc, 0) = aT; X(kPartTarget, 0) = zT; X(kPartArgmax, 0) = __int_as_float(amT);
#pragma unroll
    for (int j = 0; j < kStud; ++j) {
      X(kPartMax, j + 1) = mS[j]; X(kPartSum1, j + 1) = s1S[j]; X(kPartSumTau, j + 1) = stS[j];
      X(kPartAcc, j + 1) = aS[j]; X(kPartTarget, j + 1) = zS[j];
      X(kPartArgmax, j + 1) = __int_as_float(amS[j]);
    }
  }
  named_bar_sync(1, kHeadEpiWarps * 32);
  if (half == 1 || !row_ok) return;

  // teacher (its weighted sum is relative to its own maximum)
  const float mT1 = X(kPartMax, 0), s1T1 = X(kPartSum1, 0), stT1 = X(kPartSumTau, 0);
  const float mTm = fmaxf(mT, mT1);
  const float fa1 = scale_from(mT, mTm, L1), fb1 = scale_from(mT1, mTm, L1);
  const float fat = scale_from(mT, mTm, Lt), fbt = scale_from(mT1, mTm, Lt);
  const float accT = (mT == -INFINITY ? 0.f : fat * (aT + (mT - mTm) * Lt * stT)) +
                     (mT1 == -INFINITY ? 0.f : fbt * (X(kPartAcc, 0) + (mT1 - mTm) * Lt * stT1));
  const long long MT = static_cast<long long>(p.M) * p.T;
  MLS_CHECK(p.status, split < p.S && row < p.T);
  float* P = p.part + static_cast<long long>(split) * kPartFields * MT;
  {
    float* Pt = P + static_cast<long long>(p.order[0]) * p.T + row;
    Pt[kPartMax * MT] = mTm;
    Pt[kPartSum1 * MT] = s1T * fa1 + s1T1 * fb1;
    Pt[kPartSumTau * MT] = stT * fat + stT1 * fbt;
    Pt[kPartAcc * MT] = accT;
    Pt[kPartTarget * MT] = zT + X(kPartTarget, 0);
    Pt[kPartArgmax * MT] = __int_as_float(merged_argmax(mT, amT, mT1, __float_as_int(X(kPartArgmax, 0))));
  }
#pragma unroll
  for (int j = 0; j < kStud; ++j) {
    if (j < nst) {
      const float m1 = X(kPartMax, j + 1);
      const float mm = fmaxf(mS[j], m1);
      float* Pm = P + static_cast<long long>(p.order[j + 1]) * p.T + row;
      Pm[kPartMax * MT] = mm;
      Pm[kPartSum1 * MT] = s1S[j] * scale_from(mS[j], mm, L1) + X(kPartSum1, j + 1) * scale_from(m1, mm, L1);
      Pm[kPartSumTau * MT] = stS[j] * scale_from(mS[j], mm, Lt) + X(kPartSumTau, j + 1) * scale_from(m1, mm, Lt);
      // a student's teacher-weighted sum follows the teacher's maximum of its half
      Pm[kPartAcc * MT] = aS[j] * fat + X(kPartAcc, j + 1) * fbt;
      Pm[kPartTarget * MT] = zS[j] + X(kPartTarget, j + 1);
      Pm[kPartArgmax * MT] = __int_as_float(merged_argmax(mS[j], amS[j], m1, __float_as_int(X(kPartArgmax, j + 1))));
    }
  }
}

// ------------------------------------------------------------------ backward epilogue
template <bool kTF32>
__device__ __forceinline__ void store_chunk(void* dst, const float (&g)[32]) {
  if constexpr (kTF32) {
    float4* d = reinterpret_cast<float4*>(dst);
#pragma unroll
    for (int i = 0; i < 8; ++i) d[i] = make_float4(g[4 * i], g[4 * i + 1], g[4 * i + 2], g[4 * i + 3]);
  } else {
    uint4* d = reinterpret_cast<uint4*>(dst);
    uint32_t w[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      __nv_bfloat162 h = __floats2bfloat162_rn(g[2 * i], g[2 * i + 1]);
      w[i] = *reinterpret_cast<uint32_t*>(&h);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) d[i] = make_uint4(w[4 * i], w[4 * i + 1], w[4 * i + 2], w[4 * i + 3]);
  }
}

// Where one warp's 32x32 chunk of dL/dz goes.  bf16: staged in this warp's
// shared-memory buffers (64B swizzle: 16-byte piece j of row r sits at piece
// j ^ ((r >> 1) & 3)) and written by a TMA store; fp32: direct global stores.
struct GOut {
  const CUtensorMap* map;  // bf16 TMA store map of this sub-model
  uint32_t stage;          // this warp's two staging buffers
  uint32_t* count;         // chunks issued by this warp (buffer parity)
  int row0;                // first token row of the warp
  char* gdst;              // fp32: this thread's row pointer at the unit's first column
  bool row_ok;
};

template <bool kTF32>
__device__ __forceinline__ void put_chunk(const GOut& o, int gcol, int ch, const float (&g)[32],
                                          int lane) {
  if constexpr (kTF32) {
    if (o.row_ok) store_chunk<true>(o.gdst + ch * 32 * 4, g);
  } else {
    const uint32_t buf = o.stage + ((*o.count) & 1u) * kHeadStageChunk;
    if (lane == 0) bulk_wait_read<1>();  // the store that last used this buffer has read it
    __syncwarp();
    uint32_t w[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      __nv_bfloat162 h = __floats2bfloat162_rn(g[2 * i], g[2 * i + 1]);
      w[i] = *reinterpret_cast<uint32_t*>(&h);
    }
    const uint32_t rowaddr = buf + lane * 64;
    const uint32_t sw = (lane >> 1) & 3;
#pragma unroll
    for (int j = 0; j < 4; ++j)
      st_shared_v4(rowaddr + ((j ^ sw) << 4), w[4 * j], w[4 * j + 1], w[4 * j + 2], w[4 * j + 3]);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      // dL/dz is read back by the GEMMs only after the whole launch, so its
      // lines are the first to go from L2, ahead of the band's H and W.
      tma_store_2d_hint(o.map, buf, gcol + ch * 32, o.row0, l2_policy_evict_first());
      bulk_commit();
    }
    *o.count += 1;
  }
}

// Teacher: q = softmax(z_t / tau) (kept in q[] for the students) and
// G_t = c_t (softmax(z_t) - e_y).
template <bool kMasked, bool kTauOne, bool kTF32>
__device__ __forceinline__ void bwd_teacher(uint32_t ta, int nvalid, int yl, float L1, float Lt,
                                            float b1, float bt, float c, float (&q)[128],
                                            const GOut& o, int gcol, int lane) {
  float v[32], g[32];
#pragma unroll
  for (int ch = 0; ch < 4; ++ch) {
    tmem_ld32(ta + ch * 32, v);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const bool ok = !kMasked || (ch * 32 + i < nvalid);
      const float qv = fast_exp2(fmaf(v[i], Lt, bt));
      const float pv = kTauOne ? qv : fast_exp2(fmaf(v[i], L1, b1));
      q[ch * 32 + i] = ok ? qv : 0.f;
      g[i] = ok ? c * pv : 0.f;
    }
    const int r = yl - ch * 32;
    if (static_cast<unsigned>(r) < 32u) {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (i == r) g[i] -= c;
    }
    put_chunk<kTF32>(o, gcol, ch, g, lane);
  }
}

// Student: G_m = a1 (softmax(z_m) - e_y) + a2 (softmax(z_m / tau) - q),
// a1 = c_m (1 - alpha), a2 = c_m alpha / tau.
template <bool kMasked, bool kTauOne, bool kTF32>
__device__ __forceinline__ void bwd_student(uint32_t ta, int nvalid, int yl, float L1, float Lt,
                                            float b1, float bt, float a1, float a2,
                                            const float (&q)[128], const GOut& o, int gcol,
                                            int lane) {
  float v[32], g[32];
  const float a12 = a1 + a2;
#pragma unroll
  for (int ch = 0; ch < 4; ++ch) {
    tmem_ld32(ta + ch * 32, v);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      const bool ok = !kMasked || (ch * 32 + i < nvalid);
      const float pv = fast_exp2(fmaf(v[i], L1, b1));
      float gv;
      if (kTauOne) {
        gv = fmaf(a12, pv, -a2 * q[ch * 32 + i]);
      } else {
        const float pt = fast_exp2(fmaf(v[i], Lt, bt));
        gv = fmaf(a1, pv, a2 * (pt - q[ch * 32 + i]));
      }
      g[i] = ok ? gv : 0.f;
    }
    const int r = yl - ch * 32;
    if (static_cast<unsigned>(r) < 32u) {
#pragma unroll
      for (int i = 0; i < 32; ++i)
        if (i == r) g[i] -= a1;
    }
    put_chunk<kTF32>(o, gcol, ch, g, lane);
  }
}

template <bool kTauOne, bool kTF32>
__device__ __forceinline__ void bwd_epilogue(const HeadParams& p, uint32_t base, uint32_t tmem,
                                             int row_base, int split, int warp, int lane,
                                             volatile int* abort_flag) {
  constexpr int kElt = kTF32 ? 4 : 2;
  const int quad = warp & 3, half = warp >> 2;
  const long long row = static_cast<long long>(row_base) + quad * 32 + lane;
  const bool row_ok = row < p.T;
  const int y = row_ok ? __ldg(p.y + row) : -1;
  const bool valid = row_ok && y >= 0 && y < p.V;
  const float inv_n = *p.inv_n;
  const uint32_t tl = tmem + (static_cast<uint32_t>(quad * 32) << 16) + static_cast<uint32_t>(half * 128);
  const float L1 = p.L1, Lt = p.Ltau;
  const long long MT = static_cast<long long>(p.M) * p.T;
  const int nst = p.M - 1;
  const long long rr = row_ok ? row : 0;

  const int t = p.order[0];
  const float cT = valid ? p.coef[t] * inv_n : 0.f;
  const float bT1 = -__ldg(p.stats + static_cast<long long>(t) * p.T + rr) * L1;
  const float bTt = -__ldg(p.stats + MT + static_cast<long long>(t) * p.T + rr) * L1;
  uint32_t nchunks = 0;
  const uint32_t stage = base + HeadSmem::kStage + static_cast<uint32_t>(warp) * 2 * kHeadStageChunk;
  const int row0 = row_base + quad * 32;
  const GOut oT{&p.mapG[t], stage, &nchunks, row0,
                static_cast<char*>(p.G) + (static_cast<long long>(t) * p.g_model_stride + rr * p.g_pitch) * kElt,
                row_ok};

  float a1[kStud], a2[kStud], b1[kStud], bt[kStud];
  int ms[kStud];
#pragma unroll
  for (int j = 0; j < kStud; ++j) {
    const int m = j < nst ? p.order[j + 1] : t;
    ms[j] = m;
    const float c = valid ? p.coef[m] * inv_n : 0.f;
    a1[j] = c * p.one_minus_alpha;
    a2[j] = c * p.alpha_over_tau;
    b1[j] = -__ldg(p.stats + static_cast<long long>(m) * p.T + rr) * L1;
    bt[j] = -__ldg(p.stats + MT + static_cast<long long>(m) * p.T + rr) * L1;
  }
  float q[128];
  uint32_t acc = 0, acc_par = 0;

  for (int vt = p.vt_begin + split; vt < p.vt_end; vt += p.S) {
    const long long col0 = static_cast<long long>(vt) * kHeadBN + half * 128;
    const int nvalid = static_cast<int>(max(0LL, min(128LL, p.V - col0)));
    const int yl = y >= 0 ? static_cast<int>(y - col0) : -1;
    const int gcol = static_cast<int>(col0 - p.g_col0);  // column within the group buffer

    if (!epi_acquire(p, base, acc, acc_par, abort_flag)) break;
    {
      const uint32_t ta = tl + acc * kHeadBN;
      GOut o = oT;
      o.gdst += static_cast<long long>(gcol) * kElt;
      if (nvalid == 128)
        bwd_teacher<false, kTauOne, kTF32>(ta, 128, yl, L1, Lt, bT1, bTt, cT, q, o, gcol, lane);
      else
        bwd_teacher<true, kTauOne, kTF32>(ta, nvalid, yl, L1, Lt, bT1, bTt, cT, q, o, gcol, lane);
    }
    epi_release(base, acc, acc_par, lane);

    bool aborted = false;
#pragma unroll
    for (int j = 0; j < kStud; ++j) {
      if (j < nst && !aborted) {
        if (!epi_acquire(p, base, acc, acc_par, abort_flag)) {
          aborted = true;
          break;
        }
        const uint32_t ta = tl + acc * kHeadBN;
        const GOut o{&p.mapG[ms[j]], stage, &nchunks, row0,
                     static_cast<char*>(p.G) +
                         (static_cast<long long>(ms[j]) * p.g_model_stride + rr * p.g_pitch + gcol) * kElt,
                     row_ok};
        if (nvalid == 128)
          bwd_student<false, kTauOne, kTF32>(ta, 128, yl, L1, Lt, b1[j], bt[j], a1[j], a2[j], q,
                                             o, gcol, lane);
        else
          bwd_student<true, kTauOne, kTF32>(ta, nvalid, yl, L1, Lt, b1[j], bt[j], a1[j], a2[j], q,
                                            o, gcol, lane);
        epi_release(base, acc, acc_par, lane);
      }
    }
    if (aborted) break;
  }
  // Every staged store has finished before the CTA's shared memory goes away.
  if (!kTF32 && lane == 0) bulk_wait_all();
  __syncwarp();
}

// ------------------------------------------------------------------ kernel
template <int kMode, bool kTF32, bool kTauOne>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kHeadThreads, 1)
    head_kernel(const __grid_constant__ HeadParams p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(gbase + HeadSmem::kAbort);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + HeadSmem::kTmemSlot);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  int tt, split;
  band_unit(static_cast<int>(blockIdx.x >> 1), p.ntt, p.S, p.band, tt, split);
  const int row_base = tt * 2 * kHeadBM + static_cast<int>(rank) * kHeadBM;  // this CTA's tokens

  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int s = 0; s < kHeadStages; ++s) {
      mbar_init(HeadSmem::full(base, s), 1);
      mbar_init(HeadSmem::empty(base, s), 1);
    }
    for (uint32_t a = 0; a < 2; ++a) {
      mbar_init(HeadSmem::accf(base, a), 1);
      mbar_init(HeadSmem::acce(base, a), 2 * kHeadEpiWarps);
    }
    mbar_init(HeadSmem::drain(base), 1);
    fence_barrier_init();
  }
  if (warp == kHeadEpiWarps + 1) {
    tmem_alloc_pair(base + HeadSmem::kTmemSlot, kTmemCols);
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
      if (lane == 0) head_producer<kTF32>(p, base, row_base, rank, split, abort_flag);
    } else if (warp == kHeadEpiWarps + 1) {
      if (lane == 0 && rank == 0) head_mma<kTF32>(p, base, tmem, split, abort_flag);
      __syncwarp();
    }
  } else {
    regs_increase<kHeadEpiRegs>();
    if constexpr (kMode == kModeFwd)
      fwd_epilogue<kTauOne>(p, base, tmem, reinterpret_cast<float*>(gbase + HeadSmem::kStage),
                            row_base, split, warp, lane, abort_flag);
    else
      bwd_epilogue<kTauOne, kTF32>(p, base, tmem, row_base, split, warp, lane, abort_flag);
  }

  tc_fence_before();
  cluster_sync();
  if (warp == kHeadEpiWarps + 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, kTmemCols);
  }
}

template <int kMode>
cudaError_t launch_head(const HeadParams& p, bool tf32, bool tau_one, cudaStream_t s) {
  const int grid = 2 * p.ntt * p.S;  // CTA pairs
  if (grid <= 0) return cudaSuccess;
  const dim3 g(grid), b(kHeadThreads);
  if (tf32) {
    if (tau_one) head_kernel<kMode, true, true><<<g, b, kHeadSmem, s>>>(p);
    else head_kernel<kMode, true, false><<<g, b, kHeadSmem, s>>>(p);
  } else {
    if (tau_one) head_kernel<kMode, false, true><<<g, b, kHeadSmem, s>>>(p);
    else head_kernel<kMode, false, false><<<g, b, kHeadSmem, s>>>(p);
  }
  return cudaGetLastError();
}

template <int kMode>
cudaError_t setup_mode() {
  cudaError_t e;
#define MLS_SET(TF, TO)                                                                      \
  e = cudaFuncSetAttribute(head_kernel<kMode, TF, TO>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                           kHeadSmem);                                                       \
  if (e != cudaSuccess) return e;                                                            \
  {                                                                                          \
    cudaFuncAttributes fa;                                                                   \
    e = cudaFuncGetAttributes(&fa, head_kernel<kMode, TF, TO>);                              \
    if (e != cudaSuccess) return e;                                                          \
    if (fa.maxThreadsPerBlock < kHeadThreads || fa.numRegs != kHeadLaunchRegs)               \
      return cudaErrorLaunchOutOfResources;                                                  \
  }
  MLS_SET(true, true)
  MLS_SET(true, false)
  MLS_SET(false, true)
  MLS_SET(false, false)
#undef MLS_SET
  return cudaSuccess;
}

}  // namespace

int head_max_active_pairs() {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * 1024);
  cfg.blockDim = dim3(kHeadThreads);
  cfg.dynamicSmemBytes = kHeadSmem;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, head_kernel<kModeFwd, false, true>, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

cudaError_t launch_head_fwd(const HeadParams& p, bool tf32, bool tau_one, cudaStream_t s) {
  return launch_head<kModeFwd>(p, tf32, tau_one, s);
}
cudaError_t launch_head_bwd(const HeadParams& p, bool tf32, bool tau_one, cudaStream_t s) {
  return launch_head<kModeBwd>(p, tf32, tau_one, s);
}
cudaError_t setup_head_kernels() {
  cudaError_t e = setup_mode<kModeFwd>();
  if (e != cudaSuccess) return e;
  return setup_mode<kModeBwd>();
}

}  // namespace mls
