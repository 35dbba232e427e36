// Host side of the C ABI declared in include/mls.h: argument validation,
// workspace planning, TMA tensor-map encoding and the launch sequences of the
// forward and backward passes.  Nothing here allocates device memory.
#include <cudaTypedefs.h>

#include <climits>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <vector>

#include "mls.h"
#include "mls_kernels.h"

namespace mls {
namespace {

__device__ int g_status;  // MLS_STATUS_* bits raised by the kernels

constexpr int kMaxDevices = 64;

struct DeviceState {
  bool ready = false;
  int err = 0;
  int sms = 0;
  int gemm_pairs = 0;  // co-resident CTA pairs of the GEMM kernel
  int head_pairs = 0;  // co-resident CTA pairs of the head kernels
  int* status = nullptr;
};

std::mutex g_mu;
DeviceState g_dev[kMaxDevices];

// With MLS_DEBUG set in the environment, failures are described on stderr.
int fail(int code, const char* what, cudaError_t e = cudaSuccess) {
  static const bool verbose = std::getenv("MLS_DEBUG") != nullptr;
  if (verbose)
    std::fprintf(stderr, "[mls] %s failed: %s%s%s\n", what, e != cudaSuccess ? cudaGetErrorName(e) : "",
                 e != cudaSuccess ? " " : "", e != cudaSuccess ? cudaGetErrorString(e) : "");
  return code;
}
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

// Checks the current device once and prepares the kernels for it.
int device_state(DeviceState** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return MLS_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return MLS_ERR_DEVICE;
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceState& s = g_dev[dev];
  if (!s.ready) {
    s.ready = true;
    int major = 0, minor = 0;
    cudaError_t e;
    if ((e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&s.sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) {
      s.err = fail(MLS_ERR_CUDA, "device query", e);
    } else if (major != 10 || minor != 3) {
      s.err = fail(MLS_ERR_DEVICE, "device check (need compute capability 10.3)");
    } else if ((e = cudaGetSymbolAddress(reinterpret_cast<void**>(&s.status), g_status)) != cudaSuccess) {
      s.err = fail(MLS_ERR_CUDA, "cudaGetSymbolAddress(status)", e);
    } else if ((e = setup_head_kernels()) != cudaSuccess) {
      s.err = fail(MLS_ERR_CUDA, "head kernel attributes", e);
    } else if ((e = setup_gemm_kernels()) != cudaSuccess) {
      s.err = fail(MLS_ERR_CUDA, "gemm kernel attributes", e);
    } else if ((e = setup_eval_kernels()) != cudaSuccess) {
      s.err = fail(MLS_ERR_CUDA, "eval kernel attributes", e);
    } else if ((e = setup_spec_kernels()) != cudaSuccess) {
      s.err = fail(MLS_ERR_CUDA, "spec kernel attributes", e);
    } else if ((e = setup_junction_kernels()) != cudaSuccess) {
      s.err = fail(MLS_ERR_CUDA, "junction kernel attributes", e);
    } else if ((s.gemm_pairs = gemm_max_active_pairs()) <= 0) {
      s.err = fail(MLS_ERR_CUDA, "gemm cluster occupancy");
    } else if ((s.head_pairs = head_max_active_pairs()) <= 0) {
      s.err = fail(MLS_ERR_CUDA, "head cluster occupancy");
    } else if (!g_encode) {
      void* fn = nullptr;
      cudaDriverEntryPointQueryResult q;
      if ((e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                cudaEnableDefault, &q)) != cudaSuccess ||
          q != cudaDriverEntryPointSuccess || !fn) {
        s.err = fail(MLS_ERR_CUDA, "cuTensorMapEncodeTiled entry point", e);
      } else {
        g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
      }
    }
  }
  *out = &s;
  return s.err;
}

// Co-resident head-kernel CTA pairs on the current device, for sizing a plan
// without launching (76 on a GB300 when no device can be queried).
int current_head_pairs() {
  DeviceState* dev = nullptr;
  if (device_state(&dev) == MLS_OK && dev->head_pairs > 0) return dev->head_pairs;
  cudaGetLastError();
  return 76;
}

// ------------------------------------------------------------------ planning
constexpr size_t kAlign = 256;
size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }
long long ceil_div(long long a, long long b) { return (a + b - 1) / b; }

struct Plan {
  int elt = 2;
  int ntt = 0, nvt = 0;
  int band = 1;      // token tiles per band of the forward and evaluation launch order
  int band_bwd = 1;  // the same for the backward head kernel
  // forward
  int S = 1, nparts = 0, merge_blocks = 0, eval_merge_blocks = 0;
  size_t off_part = 0, off_bsum = 0, off_bcnt = 0, fwd_bytes = 0;
  // backward
  long long group = 0, ngroups = 0;
  size_t off_invn = 0, off_G = 0, bwd_bytes = 0;
  // fp32 inputs only: K-major copies G^T [M][group][t_pitch], H_m^T [d_m][t_pitch],
  // W_m^T [d_m][v_pitch] for the tf32 GEMMs
  long long t_pitch = 0, v_pitch = 0;
  size_t off_GT = 0, off_HT[kMaxModels] = {}, off_WT[kMaxModels] = {};
  // pairwise evaluation
  int eval_nvt = 0, eval_S = 1;
  size_t off_epart = 0, off_eacc = 0, off_ecnt = 0, eval_bytes = 0;
  size_t total = 0;
};

// CTA pairs per token tile (vocabulary splits).  Each pair of a head kernel
// walks ceil(tiles / S) vocabulary tiles and `pairs` pairs are resident at a
// time, so the kernel lasts about waves * (tiles per pair + a fixed per-pair
// cost); S minimises that.
// cta_cost: what one CTA pair costs beyond its tiles, in vocabulary tiles
// (prologue, pipeline fill and drain, the exposed epilogue of its last tile).
constexpr double kHeadCtaCost = 0.25;
// The evaluation kernel's last tile exposes its whole epilogue (every pass) and
// the partial-state write.  Measured at the 3-level suite (T = 8192, 197
// vocabulary tiles): 33 splits (the head kernels' choice) 3.39 ms per call,
// 7 splits 3.24 ms, which puts its per-pair cost near 1.2 tiles.
constexpr double kEvalCtaCost = 1.25;
int choose_splits(int ntt, long long tiles, int pairs, double cta_cost = kHeadCtaCost) {
  if (ntt < 1) ntt = 1;
  if (tiles < 1) return 1;
  long long best = 1;
  double best_cost = 1e300;
  for (long long S = 1; S <= tiles && S <= 512; ++S) {
    const long long per = (tiles + S - 1) / S;
    if (S > 1 && (per - 1) * S >= tiles) continue;  // same tiles per CTA with fewer CTAs
    const long long waves = (ntt * S + pairs - 1) / pairs;
    const double cost = waves * (per + cta_cost);
    if (cost < best_cost - 1e-9) {
      best_cost = cost;
      best = S;
    }
  }
  return static_cast<int>(best);
}

// Token tiles per band of the head kernels' launch order (band_unit): the
// pairs resident at one time re-read the hidden states of every sub-model for
// the band's tokens once per vocabulary tile, so a band's H is kept within a
// share of L2 that stays resident while W streams past it.  Fewer token tiles
// per band mean more passes over W (one per band); the bands are made equal.
// The backward streams its dL/dz stores through L2 as well, so its band's H
// gets a smaller share (measured on the 3-level suite: 48 MB gave the
// forward its least traffic at no cost in time; 32 MB, with the stores
// marked evict-first, cut the backward's DRAM reads from 4.8 to 3.3 GB).
constexpr long long kBandBytesFwd = 48ll << 20;
constexpr long long kBandBytesBwd = 32ll << 20;
int choose_band(int ntt, long long h_bytes_per_tile, long long budget) {
  if (ntt < 1) return 1;
  long long band = budget / (h_bytes_per_tile > 0 ? h_bytes_per_tile : 1);
  if (band < 1) band = 1;
  if (band >= ntt) return ntt;
  const long long nbands = (ntt + band - 1) / band;
  return static_cast<int>((ntt + nbands - 1) / nbands);
}

int validate(const mls_problem* p) {
  if (!p || p->M < 1 || p->M > MLS_MAX_MODELS || p->T < 0 || p->V < 1 || p->V > INT_MAX ||
      p->T > INT_MAX || !p->d)
    return MLS_ERR_ARG;
  if (p->teacher < 0 || p->teacher >= p->M) return MLS_ERR_ARG;
  if (!(p->tau > 0.f) || !std::isfinite(p->tau)) return MLS_ERR_ARG;
  if (!(p->alpha >= 0.f && p->alpha <= 1.f)) return MLS_ERR_ARG;
  if (p->in_dtype != MLS_BF16 && p->in_dtype != MLS_FP32) return MLS_ERR_ARG;
  if (p->vocab_group < 0 || p->vocab_group % kHeadBN != 0) return MLS_ERR_ARG;
  const int elt = p->in_dtype == MLS_BF16 ? 2 : 4;
  for (int m = 0; m < p->M; ++m) {
    if (p->d[m] < 1) return MLS_ERR_ARG;
    if ((static_cast<long long>(p->d[m]) * elt) % 16 != 0) return MLS_ERR_UNSUPPORTED;
  }
  if (p->w)
    for (int m = 0; m < p->M; ++m)
      if (!std::isfinite(p->w[m])) return MLS_ERR_ARG;
  return MLS_OK;
}

Plan make_plan(const mls_problem* p, int pairs) {
  Plan pl;
  pl.elt = p->in_dtype == MLS_BF16 ? 2 : 4;
  const long long T = p->T, V = p->V, M = p->M;
  pl.ntt = static_cast<int>(ceil_div(T, 2 * kHeadBM));  // token tiles of a CTA pair
  pl.nvt = static_cast<int>(ceil_div(V, kHeadBN));
  pl.S = choose_splits(pl.ntt, pl.nvt, pairs);
  pl.nparts = pl.S;
  long long sum_d = 0;
  for (int m = 0; m < p->M; ++m) sum_d += p->d[m];
  pl.band = choose_band(pl.ntt, 2LL * kHeadBM * sum_d * pl.elt, kBandBytesFwd);
  pl.band_bwd = choose_band(pl.ntt, 2LL * kHeadBM * sum_d * pl.elt, kBandBytesBwd);
  pl.merge_blocks = static_cast<int>(ceil_div(T, merge_tokens_per_block(pl.nparts)));
  pl.eval_merge_blocks = static_cast<int>(ceil_div(T, kEvalMergeTokens));
  size_t o = 0;
  pl.off_part = o;
  o = align_up(o + sizeof(float) * static_cast<size_t>(pl.nparts) * kPartFields * M * T);
  pl.off_bsum = o;
  o = align_up(o + sizeof(double) * static_cast<size_t>(pl.merge_blocks + 1));
  pl.off_bcnt = o;
  o = align_up(o + sizeof(long long) * static_cast<size_t>(pl.merge_blocks + 1));
  pl.fwd_bytes = o;

  // Backward vocabulary groups: the bf16 (fp32) gradient of the logits of one
  // group of columns for every sub-model stays within ~4 GiB unless the caller
  // chose the group width.
  const long long vpad = static_cast<long long>(pl.nvt) * kHeadBN;
  long long gmax = p->vocab_group;
  if (gmax == 0) {
    const long long budget = 4LL << 30;
    const long long per_col = M * (T > 0 ? T : 1) * pl.elt;
    gmax = budget / per_col / kHeadBN * kHeadBN;
    if (gmax < 2048) gmax = 2048;
  }
  if (gmax > vpad) gmax = vpad;
  pl.ngroups = ceil_div(vpad, gmax);
  pl.group = ceil_div(ceil_div(vpad, pl.ngroups), kHeadBN) * kHeadBN;
  pl.ngroups = ceil_div(vpad, pl.group);
  o = 0;
  pl.off_invn = o;
  o = align_up(o + sizeof(float));
  pl.off_G = o;
  o = align_up(o + static_cast<size_t>(pl.elt) * M * T * pl.group);
  if (pl.elt == 4) {
    pl.t_pitch = ceil_div(T, 4) * 4;
    pl.v_pitch = ceil_div(V, 4) * 4;
    pl.off_GT = o;
    o = align_up(o + sizeof(float) * static_cast<size_t>(M) * pl.group * pl.t_pitch);
    for (int m = 0; m < p->M; ++m) {
      pl.off_HT[m] = o;
      o = align_up(o + sizeof(float) * static_cast<size_t>(p->d[m]) * pl.t_pitch);
      pl.off_WT[m] = o;
      o = align_up(o + sizeof(float) * static_cast<size_t>(p->d[m]) * pl.v_pitch);
    }
  }
  pl.bwd_bytes = o;

  pl.eval_nvt = static_cast<int>(ceil_div(V, eval_tile_cols(p->M)));
  pl.eval_S = choose_splits(pl.ntt, pl.eval_nvt, pairs, kEvalCtaCost);
  o = 0;
  pl.off_epart = o;
  o = align_up(o + sizeof(float) * static_cast<size_t>(pl.eval_S) * kEvalFields * T);
  pl.off_eacc = o;
  o = align_up(o + sizeof(double) * 2 * kMaxModels * kMaxModels * static_cast<size_t>(pl.eval_merge_blocks + 1));
  pl.off_ecnt = o;
  o = align_up(o + sizeof(long long) * static_cast<size_t>(pl.eval_merge_blocks + 1));
  pl.eval_bytes = o;

  pl.total = pl.fwd_bytes > pl.bwd_bytes ? pl.fwd_bytes : pl.bwd_bytes;
  if (pl.eval_bytes > pl.total) pl.total = pl.eval_bytes;
  return pl;
}

bool aligned16(const void* ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

// 2-D row-major tensor [rows, cols] of `elt`-byte elements (128-byte swizzle
// unless told otherwise).
int encode(CUtensorMap* map, const void* ptr, int elt, long long cols, long long rows,
           long long pitch_elems, int box_cols, int box_rows,
           CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(pitch_elems) * elt};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(box_cols), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = g_encode(
      map, elt == 2 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2,
      const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
      swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
      CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    char what[160];
    std::snprintf(what, sizeof what, "cuTensorMapEncodeTiled (CUresult %d, %lld x %lld, box %d x %d)",
                  static_cast<int>(r), cols, rows, box_cols, box_rows);
    return fail(MLS_ERR_CUDA, what);
  }
  return MLS_OK;
}

void fill_head_common(HeadParams& hp, const mls_problem* p, const Plan& pl, const int* y,
                      int* status) {
  const int KE = 128 / pl.elt;
  hp.M = p->M;
  hp.order[0] = p->teacher;
  for (int m = 0, j = 1; m < p->M; ++m)
    if (m != p->teacher) hp.order[j++] = m;
  for (int m = 0; m < p->M; ++m) hp.nk[m] = static_cast<int>(ceil_div(p->d[m], KE));
  hp.ntt = pl.ntt;
  hp.T = p->T;
  hp.V = p->V;
  hp.L1 = 1.4426950408889634f;
  hp.Ltau = static_cast<float>(1.4426950408889634 / static_cast<double>(p->tau));
  hp.y = y;
  hp.status = status;
  // Failure-detection test hook: with MLS_TEST_STALL_FIRST_STAGE set, the first
  // CTA pair of a head kernel skips its first stage so that a bounded pipeline
  // wait runs out and the call reports MLS_STATUS_TIMEOUT.
  hp.test_stall = std::getenv("MLS_TEST_STALL_FIRST_STAGE") != nullptr ? 1 : 0;
}

int encode_head_maps(HeadParams& hp, const mls_problem* p, const Plan& pl, const void* const* H,
                     const void* const* W) {
  const int KE = 128 / pl.elt;
  for (int m = 0; m < p->M; ++m) {
    if (encode(&hp.mapH[m], H[m], pl.elt, p->d[m], p->T, p->d[m], KE, kHeadBM) ||
        encode(&hp.mapW[m], W[m], pl.elt, p->d[m], p->V, p->d[m], KE, kHeadBHalf))
      return MLS_ERR_CUDA;
  }
  return MLS_OK;
}

int check_ws(const Plan& pl, void* ws, size_t ws_bytes, size_t need) {
  if (need == 0) return MLS_OK;
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0 || ws_bytes < need)
    return MLS_ERR_WORKSPACE;
  return MLS_OK;
}

int launch_ok(cudaError_t e) { return e == cudaSuccess ? MLS_OK : fail(MLS_ERR_CUDA, "launch", e); }

// ------------------------------------------------------------------ kernel timing
struct ProfRec {
  const char* name;
  cudaEvent_t a, b;
};
std::mutex g_prof_mu;
bool g_prof_on = false;
std::vector<ProfRec> g_prof;
std::vector<cudaEvent_t> g_event_pool;

cudaEvent_t pool_event() {
  if (!g_event_pool.empty()) {
    cudaEvent_t e = g_event_pool.back();
    g_event_pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

// Runs `launch` (which returns a cudaError_t), bracketed by events when timing is on.
template <class F>
int timed(const char* name, cudaStream_t s, F&& launch) {
  if (!g_prof_on) return launch_ok(launch());
  std::lock_guard<std::mutex> lk(g_prof_mu);
  cudaEvent_t a = pool_event(), b = pool_event();
  if (a) cudaEventRecord(a, s);
  const int rc = launch_ok(launch());
  if (a && b) {
    cudaEventRecord(b, s);
    g_prof.push_back({name, a, b});
  }
  return rc;
}

}  // namespace
}  // namespace mls

using namespace mls;

extern "C" size_t mls_workspace_size(const mls_problem* p) {
  if (validate(p) != MLS_OK) return 0;
  return make_plan(p, current_head_pairs()).total;
}

extern "C" int mls_head_loss_fwd(const mls_problem* p, const void* const* H, const void* const* W,
                                 const int32_t* targets, float* loss, float* tok_loss,
                                 float* tok_diag, int32_t* argmax, float* stats, void* ws,
                                 size_t ws_bytes, mls_stream_t stream) {
  int rc = validate(p);
  if (rc) return rc;
  if (!H || !W || !loss || (p->T > 0 && (!targets || !tok_loss || !stats))) return MLS_ERR_ARG;
  for (int m = 0; m < p->M; ++m) {
    if ((p->T > 0 && !H[m]) || !W[m]) return MLS_ERR_ARG;  // no rows to read when T = 0
    if (!aligned16(H[m]) || !aligned16(W[m])) return MLS_ERR_ALIGN;
  }
  DeviceState* dev = nullptr;
  if ((rc = device_state(&dev))) return rc;
  const Plan pl = make_plan(p, dev->head_pairs);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (p->T == 0) return launch_ok(cudaMemsetAsync(loss, 0, sizeof(float), s));
  if ((rc = check_ws(pl, ws, ws_bytes, pl.total))) return rc;
  char* wsb = static_cast<char*>(ws);

  HeadParams hp;
  std::memset(&hp, 0, sizeof hp);
  fill_head_common(hp, p, pl, targets, dev->status);
  if ((rc = encode_head_maps(hp, p, pl, H, W))) return rc;
  hp.vt_begin = 0;
  hp.vt_end = pl.nvt;
  hp.S = pl.S;
  hp.band = pl.band;
  hp.part = reinterpret_cast<float*>(wsb + pl.off_part);
  if ((rc = timed("head_fwd", s, [&] { return launch_head_fwd(hp, pl.elt == 4, p->tau == 1.0f, s); }))) return rc;

  MergeParams mp;
  std::memset(&mp, 0, sizeof mp);
  mp.part = hp.part;
  mp.nparts = pl.nparts;
  mp.M = p->M;
  mp.teacher = p->teacher;
  mp.T = p->T;
  mp.V = p->V;
  mp.L1 = hp.L1;
  mp.Ltau = hp.Ltau;
  mp.tau = p->tau;
  mp.alpha = p->alpha;
  for (int m = 0; m < p->M; ++m) mp.w[m] = p->w ? p->w[m] : 1.0f;
  mp.y = targets;
  mp.tok_loss = tok_loss;
  mp.tok_diag = tok_diag;
  mp.argmax = argmax;
  mp.stats = stats;
  mp.block_sum = reinterpret_cast<double*>(wsb + pl.off_bsum);
  mp.block_cnt = reinterpret_cast<long long*>(wsb + pl.off_bcnt);
  mp.status = dev->status;
  if ((rc = timed("merge", s, [&] { return launch_merge(mp, pl.merge_blocks, s); }))) return rc;
  return timed("final", s, [&] { return launch_final(mp.block_sum, mp.block_cnt, pl.merge_blocks, loss, s); });
}

// The dH problems of a backward GEMM launch run in wide units
// (GemmProblem::wide) when each of them has a reduction of at least this many
// k-blocks of 128 bytes, an even number of column tiles (no single-tile
// units, which would only lose the epilogue overlap) and nothing to
// accumulate (the first vocabulary group): a wide unit's two accumulators are
// drained while no MMA runs, which costs a share inversely proportional to
// the reduction and doubles when dH is read back.  Measured on one GB300 in a
// seconds-long loop under the power cap: the 3-level suite at T = 8192 (786
// k-blocks) gains 2.6% on the GEMM, while the paper's 3B suite (9 and 17
// column tiles) lost 5% and the 4-level suite (504 k-blocks, four groups)
// 2% when they ran wide.
constexpr long long kWideMinBlocks = 512;

// Two-class schedule of a persistent GEMM launch whose first n_long tiles take
// cost_long and the other n_short cost_short (K-blocks plus a per-tile
// allowance): see GemmParams.  The pairs that get one long tile fewer take
// `catchup` short tiles first, about the cost of that long tile.
void schedule_two_class(GemmParams& g, int pairs, int n_long, long long cost_long, int n_short,
                        long long cost_short) {
  g.two_class = 0;
  if (pairs < 1 || n_long <= 0 || n_short <= 0) return;
  g.two_class = 1;
  g.n_long = n_long;
  const int r = n_long % pairs;
  int catchup = 0;
  if (r > 0) {
    catchup = static_cast<int>((cost_long + cost_short / 2) / cost_short);
    const int most = n_short / (pairs - r);
    if (catchup > most) catchup = most;
  }
  g.catchup = catchup;
}

extern "C" int mls_head_loss_bwd(const mls_problem* p, const void* const* H, const void* const* W,
                                 const int32_t* targets, const float* stats, float grad_scale,
                                 float* const* dH, float* const* dW, void* ws, size_t ws_bytes,
                                 mls_stream_t stream) {
  int rc = validate(p);
  if (rc) return rc;
  if (!H || !W || !dH || !dW || (p->T > 0 && (!targets || !stats))) return MLS_ERR_ARG;
  if (!std::isfinite(grad_scale)) return MLS_ERR_ARG;
  for (int m = 0; m < p->M; ++m) {
    if ((p->T > 0 && (!H[m] || !dH[m])) || !W[m] || !dW[m]) return MLS_ERR_ARG;
    if (!aligned16(H[m]) || !aligned16(W[m]) || !aligned16(dW[m]) || !aligned16(dH[m]))
      return MLS_ERR_ALIGN;
  }
  DeviceState* dev = nullptr;
  if ((rc = device_state(&dev))) return rc;
  const Plan pl = make_plan(p, dev->head_pairs);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (p->T == 0) {
    for (int m = 0; m < p->M; ++m)
      if ((rc = launch_ok(cudaMemsetAsync(dW[m], 0, sizeof(float) * p->V * p->d[m], s)))) return rc;
    return MLS_OK;
  }
  if ((rc = check_ws(pl, ws, ws_bytes, pl.total))) return rc;
  char* wsb = static_cast<char*>(ws);
  const bool tf32 = pl.elt == 4;
  const int KE = 128 / pl.elt;
  float* inv_n = reinterpret_cast<float*>(wsb + pl.off_invn);
  void* G = wsb + pl.off_G;

  if ((rc = timed("count", s, [&] { return launch_count(targets, p->T, p->V, inv_n, dev->status, s); }))) return rc;

  HeadParams hp;
  std::memset(&hp, 0, sizeof hp);
  fill_head_common(hp, p, pl, targets, dev->status);
  if ((rc = encode_head_maps(hp, p, pl, H, W))) return rc;
  hp.stats = stats;
  hp.inv_n = inv_n;
  for (int m = 0; m < p->M; ++m) hp.coef[m] = grad_scale * (p->w ? p->w[m] : 1.0f);
  hp.one_minus_alpha = 1.0f - p->alpha;
  hp.alpha_over_tau = p->alpha / p->tau;
  hp.G = G;
  hp.g_pitch = pl.group;
  hp.g_model_stride = p->T * pl.group;

  // bf16: dW reads A = G viewed M-major and B = H viewed N-major, dH reads
  // A = G K-major and B = W viewed N-major, all in place.
  // fp32 (tf32 MMA): dW reads A = G^T and B = H^T, dH reads A = G and B = W^T,
  // all K-major.
  GemmParams gw, gh, gb;
  std::memset(&gw, 0, sizeof gw);
  std::memset(&gh, 0, sizeof gh);
  float* GT = tf32 ? reinterpret_cast<float*>(wsb + pl.off_GT) : nullptr;
  for (int m = 0; m < p->M; ++m) {
    const void* Gm = static_cast<const char*>(G) + static_cast<size_t>(pl.elt) * hp.g_model_stride * m;
    if (encode(&gh.mapA[m], Gm, pl.elt, pl.group, p->T, pl.group, KE, kGemmBM)) return MLS_ERR_CUDA;
    // the backward head kernel's TMA stores of 32x32 dL/dz chunks (bf16 only)
    if (!tf32 && encode(&hp.mapG[m], Gm, 2, pl.group, p->T, pl.group, 32, 32,
                        CU_TENSOR_MAP_SWIZZLE_64B))
      return MLS_ERR_CUDA;
    if (!tf32) {
      if (encode(&gw.mapA[m], Gm, pl.elt, pl.group, p->T, pl.group, KE, KE) ||
          encode(&gw.mapB[m], H[m], pl.elt, p->d[m], p->T, p->d[m], KE, KE) ||
          encode(&gh.mapB[m], W[m], pl.elt, p->d[m], p->V, p->d[m], KE, KE))
        return MLS_ERR_CUDA;
    } else {
      float* HT = reinterpret_cast<float*>(wsb + pl.off_HT[m]);
      float* WT = reinterpret_cast<float*>(wsb + pl.off_WT[m]);
      if ((rc = launch_ok(launch_transpose(static_cast<const float*>(H[m]), p->T, p->d[m], p->d[m],
                                           HT, pl.t_pitch, s))) ||
          (rc = launch_ok(launch_transpose(static_cast<const float*>(W[m]), p->V, p->d[m], p->d[m],
                                           WT, pl.v_pitch, s))))
        return rc;
      if (encode(&gw.mapA[m], GT + static_cast<size_t>(m) * pl.group * pl.t_pitch, 4, p->T,
                 pl.group, pl.t_pitch, KE, kGemmBM) ||
          encode(&gw.mapB[m], HT, 4, p->T, p->d[m], pl.t_pitch, KE, kGemmBHalf) ||
          encode(&gh.mapB[m], WT, 4, p->V, p->d[m], pl.v_pitch, KE, kGemmBHalf))
        return MLS_ERR_CUDA;
    }
  }
  gw.nprob = gh.nprob = p->M;
  gw.status = gh.status = dev->status;

  const long long tiles_per_group = pl.group / kHeadBN;
  for (long long g = 0; g < pl.ngroups; ++g) {
    const long long c0 = g * pl.group;
    const long long gc = (p->V - c0 < pl.group) ? p->V - c0 : pl.group;  // columns of this group
    hp.vt_begin = static_cast<int>(g * tiles_per_group);
    hp.vt_end = static_cast<int>(ceil_div(c0 + gc, kHeadBN));
    hp.S = choose_splits(pl.ntt, hp.vt_end - hp.vt_begin, dev->head_pairs);
    hp.band = pl.band_bwd;
    hp.g_col0 = c0;
    if ((rc = timed("head_bwd", s, [&] { return launch_head_bwd(hp, tf32, p->tau == 1.0f, s); }))) return rc;
    if (tf32)
      for (int m = 0; m < p->M; ++m)
        if ((rc = launch_ok(launch_transpose(
                 reinterpret_cast<const float*>(G) + static_cast<size_t>(m) * hp.g_model_stride,
                 p->T, pl.group, pl.group, GT + static_cast<size_t>(m) * pl.group * pl.t_pitch,
                 pl.t_pitch, s))))
          return rc;

    int tw = 0, th = 0;
    for (int m = 0; m < p->M; ++m) {
      GemmProblem& a = gw.prob[m];
      a.Mrows = static_cast<int>(gc);
      a.Ncols = p->d[m];
      a.K = static_cast<int>(p->T);
      a.a_map = a.b_map = m;
      a.C = dW[m] + c0 * p->d[m];
      a.ldc = p->d[m];
      a.accumulate = 0;
      a.tiles_n = static_cast<int>(ceil_div(p->d[m], kGemmBN));
      a.tile_begin = tw;
      tw += static_cast<int>(ceil_div(gc, 2 * kGemmBM)) * a.tiles_n;

      GemmProblem& b = gh.prob[m];
      b.Mrows = static_cast<int>(p->T);
      b.Ncols = p->d[m];
      b.K = static_cast<int>(gc);
      b.a_map = b.b_map = m;
      b.b_k0 = static_cast<int>(c0);
      b.C = dH[m];
      b.ldc = p->d[m];
      b.accumulate = g > 0 ? 1 : 0;
      b.tiles_n = static_cast<int>(ceil_div(p->d[m], kGemmBN));
      b.tile_begin = th;
      th += static_cast<int>(ceil_div(p->T, 2 * kGemmBM)) * b.tiles_n;
    }
    gw.total_tiles = tw;
    gh.total_tiles = th;
    // persistent: one CTA pair per resident pair slot, never more pairs than tiles
    const int pairs = dev->gemm_pairs;
    const int grid_w = 2 * (tw < pairs ? tw : pairs), grid_h = 2 * (th < pairs ? th : pairs);
    if (tf32) {
      if ((rc = timed("gemm_dw", s, [&] { return launch_gemm_kk(gw, true, grid_w, s); }))) return rc;
      if ((rc = timed("gemm_dh", s, [&] { return launch_gemm_kk(gh, true, grid_h, s); }))) return rc;
      continue;
    }
    // bf16: dW and dH of every sub-model in one persistent launch, the class
    // with the longer reduction (dH: the group's columns, dW: T) scheduled first.
    const bool dh_long = gc >= p->T;
    const GemmParams& L = dh_long ? gh : gw;
    const GemmParams& S = dh_long ? gw : gh;
    std::memset(&gb, 0, sizeof gb);
    const int M = p->M;
    for (int m = 0; m < M; ++m) {
      gb.mapA[m] = L.mapA[m];
      gb.mapB[m] = L.mapB[m];
      gb.prob[m] = L.prob[m];
      gb.prob[m].a_map = gb.prob[m].b_map = m;
      gb.prob[m].a_mn = dh_long ? 0 : 1;
      gb.mapA[M + m] = S.mapA[m];
      gb.mapB[M + m] = S.mapB[m];
      gb.prob[M + m] = S.prob[m];
      gb.prob[M + m].a_map = gb.prob[M + m].b_map = M + m;
      gb.prob[M + m].a_mn = dh_long ? 1 : 0;
    }
    // dH with a long reduction runs in wide units (two column tiles sharing
    // each A tile of G); the units are numbered problem by problem, the long
    // class first.
    bool wide = true;
    for (int i = 0; i < 2 * M; ++i) {
      const GemmProblem& q = gb.prob[i];
      if (q.a_mn == 0)
        wide = wide && q.accumulate == 0 && q.tiles_n % 2 == 0 && ceil_div(q.K, KE) >= kWideMinBlocks;
    }
    int units = 0, n_long = 0;
    for (int i = 0; i < 2 * M; ++i) {
      GemmProblem& q = gb.prob[i];
      q.wide = (wide && q.a_mn == 0) ? 1 : 0;
      q.tile_begin = units;
      units += static_cast<int>(ceil_div(q.Mrows, 2 * kGemmBM)) * (q.wide ? (q.tiles_n + 1) / 2 : q.tiles_n);
      if (i == M - 1) n_long = units;
    }
    gb.nprob = 2 * M;
    gb.total_tiles = units;
    gb.status = dev->status;
    const int grid = 2 * (gb.total_tiles < pairs ? gb.total_tiles : pairs);
    // cost of a unit: its K-blocks (twice for a wide one) plus an allowance for
    // draining its 256x256 accumulators
    constexpr long long kDrainBlocks = 8;
    const long long cost_l = (ceil_div(gb.prob[0].K, KE) + kDrainBlocks) * (gb.prob[0].wide ? 2 : 1);
    const long long cost_s = (ceil_div(gb.prob[M].K, KE) + kDrainBlocks) * (gb.prob[M].wide ? 2 : 1);
    schedule_two_class(gb, grid / 2, n_long, cost_l, units - n_long, cost_s);
    if ((rc = timed("gemm_bwd", s, [&] { return launch_gemm_mixed(gb, grid, s); }))) return rc;
  }
  return MLS_OK;
}

extern "C" int mls_get_status(mls_stream_t stream) {
  DeviceState* dev = nullptr;
  const int rc = device_state(&dev);
  if (rc) return rc;
  if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
    return MLS_ERR_CUDA;
  int v = 0;
  if (cudaMemcpy(&v, dev->status, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess)
    return MLS_ERR_CUDA;
  const int zero = 0;
  if (cudaMemcpy(dev->status, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess)
    return MLS_ERR_CUDA;
  return v;
}

extern "C" const char* mls_strerror(int code) {
  switch (code) {
    case MLS_OK: return "success";
    case MLS_ERR_ARG: return "invalid argument";
    case MLS_ERR_ALIGN: return "device pointer not 16-byte aligned";
    case MLS_ERR_UNSUPPORTED: return "unsupported shape (row of H/W not a multiple of 16 bytes)";
    case MLS_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case MLS_ERR_CUDA: return "CUDA runtime or launch failure";
    case MLS_ERR_DEVICE: return "current device is not compute capability 10.3";
    case MLS_STATUS_BAD_TARGET: return "a target was >= V (token ignored)";
    case MLS_STATUS_TIMEOUT: return "a pipeline wait timed out; outputs are invalid";
    case MLS_STATUS_BAD_TARGET | MLS_STATUS_TIMEOUT: return "target >= V and a pipeline timeout";
    case MLS_STATUS_CHECK: return "an internal invariant failed (checked build)";
    case MLS_STATUS_DRAIN:
    case MLS_STATUS_TIMEOUT | MLS_STATUS_DRAIN:
      return "a pipeline timeout, and a shutdown wait ran out: the CUDA context is unreliable";
    default:
      return code > 0 && code < 16 ? "several status bits are set (MLS_STATUS_* in mls.h)" : "unknown code";
  }
}

extern "C" int mls_profile_enable(int on) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  g_prof_on = on != 0;
  for (auto& r : g_prof) {
    g_event_pool.push_back(r.a);
    g_event_pool.push_back(r.b);
  }
  g_prof.clear();
  return MLS_OK;
}

extern "C" int mls_profile_read(mls_kernel_time* out, int n) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (!g_prof.empty() && cudaEventSynchronize(g_prof.back().b) != cudaSuccess) return MLS_ERR_CUDA;
  int k = 0;
  const char* names[32];
  int launches[32];
  double ms[32];
  for (auto& r : g_prof) {
    float t = 0.f;
    cudaEventElapsedTime(&t, r.a, r.b);
    int i = 0;
    while (i < k && std::strcmp(names[i], r.name) != 0) ++i;
    if (i == k && k < 32) {
      names[k] = r.name;
      launches[k] = 0;
      ms[k] = 0.0;
      ++k;
    }
    if (i < 32) {
      launches[i] += 1;
      ms[i] += t;
    }
    g_event_pool.push_back(r.a);
    g_event_pool.push_back(r.b);
  }
  g_prof.clear();
  for (int i = 0; i < k && i < n; ++i) out[i] = {names[i], launches[i], ms[i]};
  return k;
}

// ------------------------------------------------------------------ forward without allocation
// Scratch for mls_head_loss_fwd_noalloc: a fixed device array that every GPU
// loading this library holds until the process exits.  Host code must not use
// the symbol's name as a device address; the address is looked up once per
// device with cudaGetSymbolAddress (that device current) and passed to the kernels.
static __device__ __align__(256) unsigned char g_noalloc_scratch[MLS_NOALLOC_SCRATCH_BYTES];

namespace mls {
namespace {
void* g_noalloc_ptr[kMaxDevices] = {};

int noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(MLS_ERR_CUDA, "cudaGetDevice", e);
  if (dev < 0 || dev >= kMaxDevices) return MLS_ERR_DEVICE;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_noalloc_ptr[dev]) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess || !ptr) return fail(MLS_ERR_CUDA, "cudaGetSymbolAddress(scratch)", e);
    g_noalloc_ptr[dev] = ptr;
  }
  *out = g_noalloc_ptr[dev];
  return MLS_OK;
}
}  // namespace
}  // namespace mls

extern "C" int mls_head_loss_fwd_noalloc(const mls_problem* p, const void* const* H,
                                         const void* const* W, const int32_t* targets, float* loss,
                                         float* tok_loss, float* tok_diag, int32_t* argmax,
                                         float* stats, mls_stream_t stream) {
  int rc = validate(p);
  if (rc) return rc;
  if (!H || !W || !loss || (p->T > 0 && (!targets || !tok_loss || !stats))) return MLS_ERR_ARG;
  for (int m = 0; m < p->M; ++m) {
    if ((p->T > 0 && !H[m]) || !W[m]) return MLS_ERR_ARG;  // no rows to read when T = 0
    if (!aligned16(H[m]) || !aligned16(W[m])) return MLS_ERR_ALIGN;
  }
  DeviceState* dev = nullptr;
  if ((rc = device_state(&dev))) return rc;
  const Plan pl = make_plan(p, dev->head_pairs);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (p->T == 0) return launch_ok(cudaMemsetAsync(loss, 0, sizeof(float), s));
  if (pl.fwd_bytes > static_cast<size_t>(MLS_NOALLOC_SCRATCH_BYTES))
    return fail(MLS_ERR_WORKSPACE, "forward needs more scratch than MLS_NOALLOC_SCRATCH_BYTES");
  void* scratch = nullptr;
  if ((rc = noalloc_scratch(&scratch))) return rc;
  char* wsb = static_cast<char*>(scratch);
  // Every word of scratch that the kernels read is written earlier in the same
  // call (partials of valid rows, one sum per merge block), so nothing is cleared.

  HeadParams hp;
  std::memset(&hp, 0, sizeof hp);
  fill_head_common(hp, p, pl, targets, dev->status);
  if ((rc = encode_head_maps(hp, p, pl, H, W))) return rc;
  hp.vt_begin = 0;
  hp.vt_end = pl.nvt;
  hp.S = pl.S;
  hp.band = pl.band;
  hp.part = reinterpret_cast<float*>(wsb + pl.off_part);
  if ((rc = timed("head_fwd", s, [&] { return launch_head_fwd(hp, pl.elt == 4, p->tau == 1.0f, s); })))
    return rc;

  MergeParams mp;
  std::memset(&mp, 0, sizeof mp);
  mp.part = hp.part;
  mp.nparts = pl.nparts;
  mp.M = p->M;
  mp.teacher = p->teacher;
  mp.T = p->T;
  mp.V = p->V;
  mp.L1 = hp.L1;
  mp.Ltau = hp.Ltau;
  mp.tau = p->tau;
  mp.alpha = p->alpha;
  for (int m = 0; m < p->M; ++m) mp.w[m] = p->w ? p->w[m] : 1.0f;
  mp.y = targets;
  mp.tok_loss = tok_loss;
  mp.tok_diag = tok_diag;
  mp.argmax = argmax;
  mp.stats = stats;
  mp.block_sum = reinterpret_cast<double*>(wsb + pl.off_bsum);
  mp.block_cnt = reinterpret_cast<long long*>(wsb + pl.off_bcnt);
  mp.status = dev->status;
  if ((rc = timed("merge", s, [&] { return launch_merge(mp, pl.merge_blocks, s); }))) return rc;
  return timed("final", s, [&] {
    return launch_final(mp.block_sum, mp.block_cnt, pl.merge_blocks, loss, s);
  });
}

extern "C" int mls_head_pairwise(const mls_problem* p, const void* const* H, const void* const* W,
                                 const int32_t* targets, float* tok_kl, int32_t* argmax,
                                 float* pair_stats, void* ws, size_t ws_bytes, mls_stream_t stream) {
  int rc = validate(p);
  if (rc) return rc;
  if (!H || !W || !pair_stats || (p->T > 0 && !tok_kl)) return MLS_ERR_ARG;
  for (int m = 0; m < p->M; ++m) {
    if ((p->T > 0 && !H[m]) || !W[m]) return MLS_ERR_ARG;  // no rows to read when T = 0
    if (!aligned16(H[m]) || !aligned16(W[m])) return MLS_ERR_ALIGN;
  }
  DeviceState* dev = nullptr;
  if ((rc = device_state(&dev))) return rc;
  const Plan pl = make_plan(p, dev->head_pairs);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (p->T == 0)
    return launch_ok(cudaMemsetAsync(pair_stats, 0, sizeof(float) * 2 * p->M * p->M, s));
  if ((rc = check_ws(pl, ws, ws_bytes, pl.total))) return rc;
  char* wsb = static_cast<char*>(ws);

  EvalParams ep;
  std::memset(&ep, 0, sizeof ep);
  const int KE = 128 / pl.elt;
  for (int m = 0; m < p->M; ++m) {
    if (encode(&ep.mapH[m], H[m], pl.elt, p->d[m], p->T, p->d[m], KE, kHeadBM) ||
        encode(&ep.mapW[m], W[m], pl.elt, p->d[m], p->V, p->d[m], KE, eval_tile_cols(p->M) / 2))
      return MLS_ERR_CUDA;
    ep.nk[m] = static_cast<int>(ceil_div(p->d[m], KE));
  }
  ep.M = p->M;
  // units of a vocabulary tile, widest sub-model first (it overlaps the epilogue)
  for (int i = 0; i < p->M; ++i) ep.order[i] = i;
  for (int i = 0; i < p->M; ++i)
    for (int k = i + 1; k < p->M; ++k)
      if (p->d[ep.order[k]] > p->d[ep.order[i]]) {
        const int t = ep.order[i];
        ep.order[i] = ep.order[k];
        ep.order[k] = t;
      }
  // Slot schedule (M = 3): the narrower of the two TMEM-slot units goes first,
  // so the epilogue's first pass runs under the longer MMAs of the other.
  if (eval_slotted(p->M)) {
    const int t = ep.order[1];
    ep.order[1] = ep.order[2];
    ep.order[2] = t;
  }
  for (int i = 0; i < p->M; ++i) ep.pos[ep.order[i]] = i;
  ep.ntt = pl.ntt;
  ep.nvt = pl.eval_nvt;
  ep.S = pl.eval_S;
  ep.band = pl.band;
  ep.T = p->T;
  ep.V = p->V;
  ep.L1 = 1.4426950408889634f;
  ep.status = dev->status;
  ep.part = reinterpret_cast<float*>(wsb + pl.off_epart);
  if ((rc = timed("pairwise", s, [&] { return launch_eval(ep, pl.elt == 4, s); }))) return rc;

  EvalMergeParams mp;
  std::memset(&mp, 0, sizeof mp);
  mp.part = ep.part;
  mp.nparts = ep.S;
  mp.M = p->M;
  mp.T = p->T;
  mp.V = p->V;
  mp.y = targets;
  mp.tok_kl = tok_kl;
  mp.argmax = argmax;
  mp.block_acc = reinterpret_cast<double*>(wsb + pl.off_eacc);
  mp.block_cnt = reinterpret_cast<long long*>(wsb + pl.off_ecnt);
  mp.status = dev->status;
  if ((rc = timed("pairwise_merge", s, [&] { return launch_eval_merge(mp, pl.eval_merge_blocks, s); })))
    return rc;
  return timed("pairwise_final", s, [&] {
    return launch_eval_final(mp.block_acc, mp.block_cnt, pl.eval_merge_blocks, p->M, pair_stats, s);
  });
}

namespace {
int junction_check(long long T, int d_prev, int d_next, int dtype, const void* const* ptrs, int n) {
  if (T < 0 || T > INT_MAX || d_prev < 1 || d_next <= d_prev) return MLS_ERR_ARG;
  if (dtype != MLS_BF16 && dtype != MLS_FP32) return MLS_ERR_ARG;
  const int elt = dtype == MLS_BF16 ? 2 : 4;
  if ((static_cast<long long>(d_prev) * elt) % 16 || (static_cast<long long>(d_next) * elt) % 16)
    return MLS_ERR_UNSUPPORTED;
  for (int i = 0; i < n; ++i) {
    if (T > 0 && !ptrs[i]) return MLS_ERR_ARG;
    if (!aligned16(ptrs[i])) return MLS_ERR_ALIGN;
  }
  return MLS_OK;
}
}  // namespace

extern "C" int mls_junction_fwd(int64_t T, int32_t d_prev, int32_t d_next, int32_t in_dtype,
                                int32_t embed_first, const void* o, const void* e, void* x,
                                mls_stream_t stream) {
  const void* ptrs[3] = {o, e, x};
  int rc = junction_check(T, d_prev, d_next, in_dtype, ptrs, 3);
  if (rc) return rc;
  DeviceState* dev = nullptr;
  if ((rc = device_state(&dev))) return rc;
  JunctionParams jp{T, d_prev, d_next, embed_first ? 1 : 0, o, e, x, nullptr, nullptr, nullptr,
                    dev->status, dev->sms};
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return timed("junction_fwd", s, [&] { return launch_junction_fwd(jp, in_dtype == MLS_FP32, s); });
}

extern "C" int mls_junction_bwd(int64_t T, int32_t d_prev, int32_t d_next, int32_t in_dtype,
                                int32_t embed_first, const void* o, const void* e, const void* g,
                                void* d_o, void* d_e, mls_stream_t stream) {
  const void* ptrs[5] = {o, e, g, d_o, d_e};
  int rc = junction_check(T, d_prev, d_next, in_dtype, ptrs, 5);
  if (rc) return rc;
  DeviceState* dev = nullptr;
  if ((rc = device_state(&dev))) return rc;
  JunctionParams jp{T, d_prev, d_next, embed_first ? 1 : 0, o, e, nullptr, g, d_o, d_e, dev->status,
                    dev->sms};
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  return timed("junction_bwd", s, [&] { return launch_junction_bwd(jp, in_dtype == MLS_FP32, s); });
}

// ------------------------------------------------------------------ speculative verify
namespace {
struct SpecPlan {
  long long Pd = 0, Pv = 0, ldz = 0, tiles = 0;
  size_t off_ev = 0, off_ed = 0, off_sv = 0, off_sd = 0, off_fv = 0, off_fd = 0;
  size_t off_stv = 0, off_std = 0, total = 0;
};

int spec_validate(const mls_spec_problem* p) {
  if (!p || p->B < 0 || p->gamma < 0 || p->V < 1 || p->V > INT_MAX) return MLS_ERR_ARG;
  if (p->in_dtype != MLS_BF16 && p->in_dtype != MLS_FP32) return MLS_ERR_ARG;
  if (static_cast<long long>(p->B) * (p->gamma + 1) > INT_MAX) return MLS_ERR_ARG;
  const int elt = p->in_dtype == MLS_BF16 ? 2 : 4;
  if (p->d_verify < 1) return MLS_ERR_ARG;
  if ((static_cast<long long>(p->d_verify) * elt) % 16 != 0) return MLS_ERR_UNSUPPORTED;
  if (!p->greedy) {
    if (p->d_draft < 1) return MLS_ERR_ARG;
    if ((static_cast<long long>(p->d_draft) * elt) % 16 != 0) return MLS_ERR_UNSUPPORTED;
    if (!(p->temperature > 0.f) || !std::isfinite(p->temperature)) return MLS_ERR_ARG;
    if (!(p->top_p > 0.f && p->top_p <= 1.f)) return MLS_ERR_ARG;
    if (p->V > static_cast<long long>(kSpecMaxTiles) * kGemmBN || p->gamma > kSpecMaxGamma)
      return MLS_ERR_UNSUPPORTED;
  }
  return MLS_OK;
}

SpecPlan spec_plan(const mls_spec_problem* p) {
  SpecPlan pl;
  pl.Pv = static_cast<long long>(p->B) * (p->gamma + 1);
  pl.Pd = p->greedy ? 0 : static_cast<long long>(p->B) * p->gamma;
  pl.ldz = ceil_div(p->V, 4) * 4;
  pl.tiles = ceil_div(p->V, kGemmBN);
  const size_t rows_e = p->greedy ? 0 : static_cast<size_t>(pl.Pv);  // e_t is only stored when sampling
  size_t o = 0;
  auto take = [&](size_t& off, size_t bytes) {
    off = o;
    o = align_up(o + bytes);
  };
  take(pl.off_ev, sizeof(float) * rows_e * pl.ldz);
  take(pl.off_ed, sizeof(float) * static_cast<size_t>(pl.Pd) * pl.ldz);
  take(pl.off_stv, sizeof(float) * 2 * static_cast<size_t>(pl.Pv) * pl.tiles);
  take(pl.off_std, sizeof(float) * 2 * static_cast<size_t>(pl.Pd) * pl.tiles);
  take(pl.off_fv, sizeof(float) * rows_e * pl.tiles);
  take(pl.off_fd, sizeof(float) * static_cast<size_t>(pl.Pd) * pl.tiles);
  take(pl.off_sv, sizeof(float) * kSpecStateWords * static_cast<size_t>(pl.Pv));
  take(pl.off_sd, sizeof(float) * kSpecStateWords * static_cast<size_t>(pl.Pd));
  pl.total = o;
  return pl;
}
}  // namespace

extern "C" size_t mls_spec_workspace_size(const mls_spec_problem* p) {
  if (spec_validate(p)) return 0;
  return spec_plan(p).total;
}

extern "C" int mls_spec_verify(const mls_spec_problem* p, const void* H_draft, const void* W_draft,
                               const void* H_verify, const void* W_verify,
                               const int32_t* draft_tokens, const float* uniforms,
                               int32_t* n_accepted, int32_t* next_token, void* ws, size_t ws_bytes,
                               mls_stream_t stream) {
  int rc = spec_validate(p);
  if (rc) return rc;
  if (p->B == 0) return MLS_OK;
  if (!H_verify || !W_verify || !n_accepted || !next_token || (p->gamma > 0 && !draft_tokens))
    return MLS_ERR_ARG;
  if (!p->greedy && (!uniforms || (p->gamma > 0 && (!H_draft || !W_draft)))) return MLS_ERR_ARG;
  if (!aligned16(H_verify) || !aligned16(W_verify) || !aligned16(H_draft) || !aligned16(W_draft))
    return MLS_ERR_ALIGN;
  const SpecPlan pl = spec_plan(p);
  if (!ws || (reinterpret_cast<uintptr_t>(ws) % kAlign) != 0 || ws_bytes < pl.total)
    return MLS_ERR_WORKSPACE;
  DeviceState* dev = nullptr;
  if ((rc = device_state(&dev))) return rc;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  char* wsb = static_cast<char*>(ws);
  const bool tf32 = p->in_dtype == MLS_FP32;
  const int elt = tf32 ? 4 : 2, KE = 128 / elt;
  auto at = [&](size_t off) { return reinterpret_cast<float*>(wsb + off); };

  SpecParams sp;
  std::memset(&sp, 0, sizeof sp);
  sp.V = p->V;
  sp.ldz = pl.ldz;
  sp.B = p->B;
  sp.gamma = p->gamma;
  sp.greedy = p->greedy ? 1 : 0;
  sp.tiles = static_cast<int>(pl.tiles);
  sp.scale = p->greedy ? 1.f : 1.4426950408889634f / p->temperature;
  sp.top_p = p->greedy ? 1.f : p->top_p;
  sp.ev = at(pl.off_ev);
  sp.ed = at(pl.off_ed);
  sp.stats_v = at(pl.off_stv);
  sp.stats_d = at(pl.off_std);
  sp.f_v = at(pl.off_fv);
  sp.f_d = at(pl.off_fd);
  sp.draft = draft_tokens;
  sp.u = uniforms;
  sp.state_v = at(pl.off_sv);
  sp.state_d = at(pl.off_sd);
  sp.n_accepted = n_accepted;
  sp.next_token = next_token;
  sp.status = dev->status;

  // Logits of the verify positions: one GEMM launch over the verifier's rows
  // and (sampling) the draft's, z = H W^T with both operands K-major; its
  // epilogue leaves per-tile softmax statistics (sampling) or the per-tile
  // maximum and argmax (greedy) instead of the logits.
  GemmParams g;
  std::memset(&g, 0, sizeof g);
  const void* Hs[2] = {H_verify, H_draft};
  const void* Ws[2] = {W_verify, W_draft};
  const int ds[2] = {p->d_verify, p->d_draft};
  const long long Ps[2] = {pl.Pv, pl.Pd};
  float* Cs[2] = {at(pl.off_ev), at(pl.off_ed)};
  float* Ss[2] = {at(pl.off_stv), at(pl.off_std)};
  int tiles = 0;
  for (int m = 0; m < 2; ++m) {
    if (Ps[m] == 0) continue;
    const int i = g.nprob++;
    if (encode(&g.mapA[i], Hs[m], elt, ds[m], Ps[m], ds[m], KE, kGemmBM) ||
        encode(&g.mapB[i], Ws[m], elt, ds[m], p->V, ds[m], KE, kGemmBHalf) ||
        (!p->greedy && encode(&g.mapC[i], Cs[m], 4, p->V, Ps[m], pl.ldz, 32, 32)))
      return MLS_ERR_CUDA;
    GemmProblem& pr = g.prob[i];
    pr.Mrows = static_cast<int>(Ps[m]);
    pr.Ncols = static_cast<int>(p->V);
    pr.K = ds[m];
    pr.a_map = pr.b_map = i;
    pr.C = Cs[m];
    pr.ldc = pl.ldz;
    pr.tiles_n = static_cast<int>(pl.tiles);
    pr.tiles_m = static_cast<int>(ceil_div(Ps[m], 2 * kGemmBM));
    pr.m_fast = 1;
    pr.tile_begin = tiles;
    pr.epi = p->greedy ? kEpiArgmax : kEpiSoftmax;
    pr.epi_scale = sp.scale;
    pr.stats = Ss[m];
    pr.stats_ld = 2 * pl.tiles;
    tiles += pr.tiles_m * pr.tiles_n;
  }
  g.total_tiles = tiles;
  g.status = dev->status;
  const int grid = 2 * (tiles < dev->gemm_pairs ? tiles : dev->gemm_pairs);
  if ((rc = timed("spec_logits", s, [&] { return launch_gemm_stats(g, tf32, grid, s); }))) return rc;
  if (!p->greedy && (rc = timed("spec_rows", s, [&] { return launch_spec_rows(sp, s); })))
    return rc;
  return timed("spec_sample", s, [&] { return launch_spec_sample(sp, s); });
}
