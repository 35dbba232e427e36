// Internal interface between the host API (mls_api.cu) and the kernel
// translation units.  Parameter blocks are passed by value as __grid_constant__
// kernel arguments, so the tensor maps live in the kernel parameter space.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace mls {

constexpr int kMaxModels = 4;

// ------------------------------------------------------------------ head kernels
// A CTA pair owns 2 x kHeadBM tokens and walks vocabulary tiles of kHeadBN
// columns; for each vocabulary tile it computes the teacher's logit tile first
// and then every student's, all into TMEM (double-buffered).  Each CTA holds
// its kHeadBM token rows and kHeadBHalf vocabulary rows per stage.
constexpr int kHeadBM = 128;
constexpr int kHeadBN = 256;
constexpr int kHeadBHalf = 128;
constexpr int kHeadStages = 6;
constexpr int kHeadEpiWarps = 8;                       // warpgroups 0 and 1
constexpr int kHeadThreads = (kHeadEpiWarps + 4) * 32;  // + warpgroup 2: TMA, MMA, 2 idle
// Registers: launched at 168 per thread (384 x 168 = 64512), then the control
// warpgroup gives up registers and the epilogue warpgroups take them:
// 2 x 128 x 232 + 128 x 40 = 64512.  Per SM sub-partition: 232 + 232 + 40 warps' worth.
constexpr int kHeadLaunchRegs = 168;
constexpr int kHeadEpiRegs = 232;
constexpr int kHeadCtlRegs = 40;
static_assert(2 * 128 * kHeadEpiRegs + 128 * kHeadCtlRegs == kHeadThreads * kHeadLaunchRegs,
              "register reallocation must add up to the launch allocation");
constexpr uint32_t kHeadABytes = kHeadBM * 128;
constexpr uint32_t kHeadBBytes = kHeadBHalf * 128;
// Backward: each epilogue warp stages its dL/dz chunks (32 tokens x 32 bf16
// columns, 2 KB, 64B-swizzled) in two buffers and writes them with TMA stores.
constexpr uint32_t kHeadStageChunk = 32 * 64;
constexpr uint32_t kHeadStaging = kHeadEpiWarps * 2 * kHeadStageChunk;
constexpr uint32_t kHeadSmem = kHeadStages * (kHeadABytes + kHeadBBytes) + kHeadStaging + 1024 + 1024;

// Token tile and vocabulary split of CTA pair `pair` in a head or evaluation
// launch of ntt x S pairs.  Pairs are numbered band by band: a band is `band`
// consecutive token tiles (the last one may be shorter) and all S splits of
// them, token tile fastest.  The hardware starts clusters roughly in index
// order, so the pairs resident at one time cover the token tiles of one band
// and a few consecutive splits: the hidden states they re-read for every
// vocabulary tile are the band's, and each vocabulary tile is fetched by all
// the band's token tiles at about the same time.  band >= ntt gives the plain
// token-fastest order over all token tiles.
__host__ __device__ inline void band_unit(int pair, int ntt, int S, int band, int& tt, int& split) {
  if (band < 1 || band > ntt) band = ntt;
  const int per_band = band * S;
  const int b = pair / per_band;
  const int i = pair - b * per_band;
  const int nb = ntt - b * band < band ? ntt - b * band : band;
  tt = b * band + i % nb;
  split = i / nb;
}

// Partial row state written by the forward head kernel, per (partial, field, model, token).
// kPartAcc holds, for a student, sum_v q~_v z_m[v] with q~ relative to the
// teacher's running maximum of the same partial; for the teacher,
// sum_v q~_v (z_t[v] - max_t) log2(e) / tau.
enum PartField { kPartMax = 0, kPartSum1, kPartSumTau, kPartAcc, kPartTarget, kPartArgmax, kPartFields };

struct HeadParams {
  CUtensorMap mapH[kMaxModels];  // H_m [T, d_m], box {128 B of K, kHeadBM rows}
  CUtensorMap mapW[kMaxModels];  // W_m [V, d_m], box {128 B of K, kHeadBN rows}
  int M;
  int order[kMaxModels];         // order[0] = teacher, then the students
  int nk[kMaxModels];            // k-blocks (128 bytes of K each) of model m
  int ntt;                       // token tiles of 2 * kHeadBM (one per CTA pair)
  int vt_begin, vt_end;          // vocabulary tiles handled by this launch
  int S;                         // CTAs per token tile (vocabulary splits)
  int band;                      // token tiles per band of the launch order (band_unit)
  long long T, V;
  float L1;                      // log2(e)
  float Ltau;                    // log2(e) / tau
  const int* y;                  // targets [T]
  int* status;
  int test_stall;                // test hook: see head_producer (0 in normal use)
  // forward
  float* part;                   // [S][kPartFields][M][T]
  // backward
  const float* stats;            // [2][M][T]: logsumexp(z), logsumexp(z/tau)
  const float* inv_n;            // device scalar 1/N (0 if N == 0)
  float coef[kMaxModels];        // grad_scale * w_m
  float one_minus_alpha;         // (1 - alpha)
  float alpha_over_tau;          // alpha / tau
  CUtensorMap mapG[kMaxModels];  // G_m [T, g_pitch] bf16, box {32, 32}, 64B swizzle (TMA store)
  void* G;                       // [M][T][g_pitch] bf16 (fp32 for fp32 inputs)
  long long g_model_stride;      // elements
  long long g_pitch;             // elements per token row
  long long g_col0;              // vocabulary column of the group's first column
};

// ------------------------------------------------------------------ GEMM kernels
// CTA pairs: a pair owns a 256 x kGemmBN output tile; each CTA of the pair
// holds 128 rows of A and kGemmBHalf rows of B per stage.
constexpr int kGemmBM = 128;       // rows of A (and of C) per CTA
constexpr int kGemmBN = 256;       // columns of C per pair tile
constexpr int kGemmBHalf = 128;    // rows of B per CTA
constexpr int kGemmStages = 6;
// Wide units (GemmProblem::wide): stages of A | B0 | B1 over the same memory.
constexpr int kGemmWideStages = 4;
constexpr int kGemmEpiWarps = 4;
constexpr int kGemmThreads = (kGemmEpiWarps + 2) * 32;
constexpr uint32_t kGemmABytes = kGemmBM * 128;
constexpr uint32_t kGemmBBytes = kGemmBHalf * 128;
// 32 KB of slack past the last stage keeps every operand read of a descriptor
// inside the CTA's allocation.
constexpr uint32_t kGemmSmem = kGemmStages * (kGemmABytes + kGemmBBytes) + 1024 + 1024 + 32768;

struct GemmProblem {
  int Mrows, Ncols, K;           // C is Mrows x Ncols, reduction length K
  int a_map, b_map;              // index into mapA / mapB
  int a_m0, a_k0, b_n0, b_k0;    // coordinate offsets into the tensors
  float* C;                      // row-major fp32, leading dimension ldc
  long long ldc;
  int accumulate;                // C += A*B if 1, C = A*B if 0
  int tiles_n;                   // ceil(Ncols / kGemmBN)
  int tile_begin;                // first unit of this problem in the launch's unit numbering
                                 // (a unit is one pair tile of 256 x kGemmBN, or two if wide)
  int tiles_m;                   // ceil(Mrows / 256); used when m_fast is set
  int m_fast;                    // 1: consecutive tiles walk M first (pairs running at the
                                 //    same time share the B tile, read once from HBM)
  // Epilogue (accumulate must be 0 unless kEpiPlain).  Per row and column tile
  // (kGemmBN columns) the statistics go to stats[row * stats_ld + 2 * tile]:
  //   kEpiSoftmax: C = 2^((z - m_t) epi_scale), stats = (m_t, sum of C over the tile)
  //   kEpiArgmax:  C untouched, stats = (m_t, first column attaining m_t)
  // with m_t the row's maximum over the tile.
  int epi;
  float epi_scale;
  float* stats;
  long long stats_ld;
  int a_mn;                      // A is MN-major (read by launches that take the layout per problem)
  // Wide units (launch_gemm_mixed only): a unit is two adjacent column tiles
  // (tn, tn + 1) that share the A tile of each stage and take both TMEM
  // accumulators, which halves the A operand's shared-memory traffic per FLOP
  // and the number of passes over B.  The accumulators are then not double
  // buffered, so this suits problems with a long reduction.
  int wide;
};
enum GemmEpilogue { kEpiPlain = 0, kEpiSoftmax = 1, kEpiArgmax = 2 };

constexpr int kGemmMaxProblems = 2 * kMaxModels;

struct GemmParams {
  CUtensorMap mapA[kGemmMaxProblems];
  CUtensorMap mapB[kGemmMaxProblems];
  CUtensorMap mapC[kGemmMaxProblems];  // kEpiSoftmax: C fp32 [Mrows, Ncols], box {32, 32}, 128B swizzle
  int nprob;
  GemmProblem prob[kGemmMaxProblems];
  int total_tiles;               // units of the launch (pair tiles, or pairs of them if wide)
  int* status;
  // Schedule.  two_class == 0: pair p takes tiles p, p + npairs, ...
  // two_class == 1: tiles [0, n_long) are the long ones (larger K) and go
  // round-robin first, so the first r = n_long % npairs pairs get one more.
  // The other pairs then take `catchup` short tiles each, round-robin among
  // themselves, to even out that extra long tile; the remaining short tiles go
  // round-robin over all pairs.  Neighbouring tiles (which share operands in
  // L2) keep running at the same time.
  int two_class;
  int n_long;
  int catchup;
};

// ------------------------------------------------------------------ pairwise evaluation
// Forward-only evaluation metrics between sub-models.  A CTA pair owns 256
// tokens; for every vocabulary tile it computes the logit tiles of all M <= 4
// sub-models and accumulates, for every ordered pair (s, j),
// D_sj = sum_v exp(z_s[v] - max_s) (z_s[v] - z_j[v]), which needs every
// sub-model's logit at the same column.  Operand bytes per FLOP fall as the
// tile widens, and operand delivery from L2 bounds this kernel, so the tile is
// as wide as the 512 TMEM columns and the epilogue's registers allow:
//   - M = 1, 2, 4: all M tiles resident in TMEM at once (256, 256, 128 columns);
//   - M = 3 (eval_slotted): 256 columns; the widest sub-model's tile is copied
//     into the epilogue's registers as soon as it is complete, the other two
//     occupy two 256-column TMEM slots whose roles alternate from tile to tile.
__host__ __device__ constexpr bool eval_slotted(int M) { return M == 3; }
__host__ __device__ constexpr int eval_tile_cols(int M) { return M <= 3 ? 256 : 128; }
constexpr uint32_t kEvalABytes = kHeadBM * 128;                    // A stage: 128 token rows
__host__ __device__ constexpr uint32_t eval_b_bytes(int M) { return eval_tile_cols(M) / 2 * 128; }
// As many stages as fit in 216 KB (9 for M = 4, 6 for M = 1, 2, 3).
constexpr uint32_t kEvalStageBudget = 216 * 1024;
__host__ __device__ constexpr int eval_stages(int M) {
  return static_cast<int>(kEvalStageBudget / (kEvalABytes + eval_b_bytes(M)));
}
__host__ __device__ constexpr uint32_t eval_smem(int M) {
  return static_cast<uint32_t>(eval_stages(M)) * (kEvalABytes + eval_b_bytes(M)) + 1024 + 1024;
}
// per token and split: max_s (4), sum_s (4), argmax_s (4), D_sj for j != s (4 x 3)
constexpr int kEvalFields = 24;
constexpr uint32_t kEvalXchg = kEvalFields * kHeadBM * 4;
// The half-merge exchange is only used after the main loop, when the operand
// stages are idle, so it shares their memory.
static_assert(kEvalXchg <= 6 * (kEvalABytes + eval_b_bytes(2)), "exchange fits in the stages");

struct EvalParams {
  CUtensorMap mapH[kMaxModels];  // H_m [T, d_m], box {128 B of K, kHeadBM rows}
  CUtensorMap mapW[kMaxModels];  // W_m [V, d_m], box {128 B of K, eval_tile_cols(M) / 2 rows}
  int M;
  int order[kMaxModels];         // units of a vocabulary tile, widest sub-model first (M = 3:
                                 // widest, narrowest, middle)
  int pos[kMaxModels];           // pos[order[i]] = i
  int nk[kMaxModels];
  int ntt;                       // token tiles of 256 (one per CTA pair)
  int nvt;                       // vocabulary tiles of eval_tile_cols(M) columns
  int S;                         // CTA pairs per token tile
  int band;                      // token tiles per band of the launch order (band_unit)
  long long T, V;
  float L1;
  int* status;
  float* part;                   // [S][kEvalFields][T]
};

struct EvalMergeParams {
  const float* part;
  int nparts, M;
  long long T, V;
  const int* y;                  // may be null: every token counts
  float* tok_kl;                 // [M][M][T]
  int* argmax;                   // [M][T] or null
  double* block_acc;             // [blocks][2][M*M]: sums of KL and of agreement
  long long* block_cnt;          // [blocks]
  int* status;
};

// ------------------------------------------------------------------ junction (Eq. 1)
struct JunctionParams {
  long long T;
  int d_prev, d_next;            // D_m and D_{m+1}
  int embed_first;               // 0: x = [o~, e]; 1: x = [e, o~]
  const void* o;                 // [T, D_m]
  const void* e;                 // [T, D_{m+1} - D_m]
  void* x;                       // [T, D_{m+1}] (forward)
  const void* g;                 // [T, D_{m+1}] (backward)
  void* d_o;                     // [T, D_m] (backward)
  void* d_e;                     // [T, D_{m+1} - D_m] (backward)
  int* status;                   // device status word (pipeline-wait timeouts)
  int sms;                       // SMs of the device
};
cudaError_t launch_junction_fwd(const JunctionParams& p, bool fp32, cudaStream_t s);
cudaError_t launch_junction_bwd(const JunctionParams& p, bool fp32, cudaStream_t s);
cudaError_t setup_junction_kernels();

// ------------------------------------------------------------------ speculative verify
// Per position of a sequence: the verifier's logits row (and the draft's for
// the gamma drafted positions), fp32 with row pitch ldz (a multiple of 4).
// The logits GEMM's epilogue leaves, per row, e_t[v] = 2^((z[v] - m_t) log2(e) / T)
// relative to the maximum m_t of v's column tile, and per tile (m_t, sum of e_t)
// (kEpiSoftmax); greedy verification only needs per tile (m_t, argmax) (kEpiArgmax).
constexpr int kSpecStateWords = 8;    // per row: max, b, kept mass, c, ties, sum (+2 spare)
constexpr int kSpecListCap = 4096;    // candidates per shared-memory list (two lists)
constexpr int kSpecMaxTiles = 4096;   // column tiles of a row (V <= 4096 * kGemmBN when sampling)
constexpr int kSpecMaxGamma = 1024;   // drafted tokens per sequence when sampling

struct SpecParams {
  long long V, ldz;
  int B, gamma;
  int greedy;
  int tiles;                     // column tiles of kGemmBN per row
  float scale;                   // log2(e) / temperature
  float top_p;
  const float* ed;               // [B * gamma][ldz] draft e_t (sampling only)
  const float* ev;               // [B * (gamma + 1)][ldz] verifier e_t (sampling only)
  const float* stats_d;          // [B * gamma][tiles][2]
  const float* stats_v;          // [B * (gamma + 1)][tiles][2]
  float* f_d;                    // [B * gamma][tiles]: 2^((m_t - max) log2(e) / T)
  float* f_v;                    // [B * (gamma + 1)][tiles]
  const int* draft;              // [B * gamma]
  const float* u;                // [B][gamma + 1][2]
  float* state_d;                // [B * gamma][kSpecStateWords]
  float* state_v;                // [B * (gamma + 1)][kSpecStateWords]
  int* n_accepted;               // [B]
  int* next_token;               // [B]
  int* status;                   // checked build: invariant failures
};
cudaError_t setup_spec_kernels();
cudaError_t launch_spec_rows(const SpecParams& p, cudaStream_t s);
cudaError_t launch_spec_sample(const SpecParams& p, cudaStream_t s);

// ------------------------------------------------------------------ reductions
struct MergeParams {
  const float* part;             // [nparts][kPartFields][M][T]
  int nparts;
  int M, teacher;
  long long T, V;
  float L1, Ltau, tau, alpha;
  float w[kMaxModels];
  const int* y;
  float* tok_loss;               // [M][T]
  float* tok_diag;               // [3][M][T] or nullptr
  int* argmax;                   // [M][T] or nullptr
  float* stats;                  // [2][M][T]
  double* block_sum;             // [gridDim.x]: sum over the block's tokens of sum_m w_m L_m
  long long* block_cnt;          // [gridDim.x]: valid tokens in the block
  int* status;
};

// Warps of a merge block per group of 8 tokens: 4 partial slots per warp, as
// few warps as cover the partials (8 warps for more than 8 partials).
__host__ __device__ inline int merge_warps_per_octet(int nparts) {
  return nparts <= 4 ? 1 : nparts <= 8 ? 2 : 8;
}
// Tokens per merge block (8 warps): 8 octets of one warp, 4 of two, or 1 of eight.
__host__ __device__ inline int merge_tokens_per_block(int nparts) {
  return 8 * (8 / merge_warps_per_octet(nparts));
}
constexpr int kEvalMergeTokens = 128;  // tokens per evaluation-merge block: one thread per token

// Launchers (return the cudaError_t of the launch).
cudaError_t launch_head_fwd(const HeadParams& p, bool tf32, bool tau_one, cudaStream_t s);
cudaError_t launch_head_bwd(const HeadParams& p, bool tf32, bool tau_one, cudaStream_t s);
// bf16, B MN-major, A's layout per problem (GemmProblem::a_mn): dW and dH in one launch.
cudaError_t launch_gemm_mixed(const GemmParams& p, int grid, cudaStream_t s);
// Both operands K-major (tf32 path: fp32 inputs with transposed copies);
// plain epilogues only.
cudaError_t launch_gemm_kk(const GemmParams& p, bool tf32, int grid, cudaStream_t s);
// Both operands K-major, with the statistics epilogues (GemmProblem::epi).
cudaError_t launch_gemm_stats(const GemmParams& p, bool tf32, int grid, cudaStream_t s);
cudaError_t launch_transpose(const float* in, long long rows, long long cols, long long ld_in,
                             float* out, long long ld_out, cudaStream_t s);
cudaError_t launch_merge(const MergeParams& p, int blocks, cudaStream_t s);
cudaError_t launch_final(const double* block_sum, const long long* block_cnt, int nblocks,
                         float* loss, cudaStream_t s);
cudaError_t launch_count(const int* y, long long T, long long V, float* inv_n, int* status,
                         cudaStream_t s);

cudaError_t launch_eval(const EvalParams& p, bool tf32, cudaStream_t s);
cudaError_t launch_eval_merge(const EvalMergeParams& p, int blocks, cudaStream_t s);
cudaError_t launch_eval_final(const double* block_acc, const long long* block_cnt, int nblocks,
                              int M, float* pair_stats, cudaStream_t s);
cudaError_t setup_eval_kernels();

// One-time per-device kernel attribute setup (dynamic shared memory limits).
cudaError_t setup_head_kernels();
cudaError_t setup_gemm_kernels();
int gemm_max_active_pairs();  // 0 if the query failed
int head_max_active_pairs();

}  // namespace mls
