/*
 * mls.h -- C ABI of the fused Matryoshka-suite output stage on GB300 (sm_103a).
 *
 * The operation (paper: "Matryoshka Language Model Suites", Sec. 2):
 *   for every nested sub-model m = 0..M-1 with hidden states H_m [T, d_m] and
 *   LM head W_m [V, d_m] (Sec. 2, "Inter-model Junction": W^m in R^{V x D_m}),
 *     z_m    = H_m W_m^T                                    (never stored)
 *     CE_m   = logsumexp(z_m) - z_m[y]                      (Sec. 2, "Modeling")
 *     Ld_m   = -sum_v q_v log softmax(z_m / tau)_v,  q = stop_grad(softmax(z_t / tau))
 *              with t the teacher sub-model                 (Eq. 2)
 *     L_m    = (1 - alpha) CE_m + alpha Ld_m  for m != t;  L_t = CE_t   (Eq. 3)
 *     loss   = sum_m w_m (1/N) sum_{tokens with y >= 0} L_m           (sum after Eq. 3, App. G)
 *   and its gradients dH_m, dW_m (teacher distribution under stop-gradient).
 *   tau is an extension: Eq. 2 is the case tau = 1.  The [T, V] logits of a
 *   sub-model are never written to memory.
 *
 * Conventions shared by every entry point:
 *   - Pointer arguments named H, W, targets, loss, tok_loss, tok_diag, argmax,
 *     stats, dH, dW and ws are DEVICE pointers owned by the caller; the arrays
 *     H, W, dH, dW themselves (the pointer lists, length M) and everything in
 *     mls_problem are HOST memory read during the call only.
 *   - All matrices are row-major and dense: H_m has row pitch d_m elements,
 *     W_m row pitch d_m, dH_m and dW_m row pitch d_m floats.  H_m and W_m must be
 *     16-byte aligned and d_m * sizeof(element) a multiple of 16 bytes.
 *   - Calls are asynchronous on `stream`; nothing is allocated and the host
 *     never synchronises.  The caller provides a workspace of at least
 *     mls_workspace_size() bytes (256-byte aligned); its contents need not be
 *     preserved between calls.
 *   - Return value: 0 on success or a negative MLS_ERR_* code, in which case
 *     nothing was launched.  Conditions only the device can see (a target >= V,
 *     an internal wait that timed out) are recorded in a status word read by
 *     mls_get_status().
 */
#ifndef MLS_H
#define MLS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* mls_stream_t;

/* Storage type of H and W.  Outputs are always fp32. */
enum { MLS_BF16 = 0, MLS_FP32 = 1 };

/* Return codes (negative) and status bits (positive, from mls_get_status). */
enum {
  MLS_OK = 0,
  MLS_ERR_ARG = -1,          /* null pointer, size or parameter out of range */
  MLS_ERR_ALIGN = -2,        /* a device pointer breaks the alignment rules above */
  MLS_ERR_UNSUPPORTED = -3,  /* shape the kernels do not handle (see mls_problem) */
  MLS_ERR_WORKSPACE = -4,    /* workspace NULL, misaligned or smaller than required */
  MLS_ERR_CUDA = -5,         /* a CUDA runtime call or kernel launch failed */
  MLS_ERR_DEVICE = -6,       /* current device is not a compute-capability 10.3 GPU */
  MLS_STATUS_BAD_TARGET = 1, /* some target was >= V; that token was treated as ignored */
  MLS_STATUS_TIMEOUT = 2,    /* a pipeline wait exceeded its bound; outputs are invalid */
  MLS_STATUS_CHECK = 4,      /* checked build only: an internal invariant failed */
  MLS_STATUS_DRAIN = 8       /* after a timeout, a kernel's bounded shutdown wait for its own
                                copies or MMAs also ran out: some may still have been in flight
                                when it exited, so the CUDA context should not be trusted */
};

/* Maximum number of sub-models per call. */
#define MLS_MAX_MODELS 4

typedef struct {
  int32_t M;            /* sub-models, 1..MLS_MAX_MODELS */
  int64_t T;            /* tokens, >= 0 */
  int64_t V;            /* vocabulary size, 1 .. 2^31 - 1 */
  const int32_t* d;     /* host array [M]: width d_m of sub-model m (> 0) */
  int32_t teacher;      /* distillation teacher, 0..M-1 (paper: M-1, the largest) */
  float tau;            /* distillation temperature > 0 (paper: 1) */
  float alpha;          /* alpha_d of Eq. 3, in [0, 1] */
  const float* w;       /* host array [M] of loss weights (App. G), or NULL for all 1 */
  int32_t in_dtype;     /* MLS_BF16 or MLS_FP32: storage type of every H_m and W_m */
  int64_t vocab_group;  /* backward vocabulary group (columns), multiple of 256, or 0 = automatic */
} mls_problem;

/*
 * Bytes of device workspace that mls_head_loss_fwd, mls_head_loss_bwd and
 * mls_head_pairwise need for this problem (the largest of the three).  Returns 0 if the problem is
 * invalid.  The backward keeps the gradient of the logits for one vocabulary
 * group, bf16 [M, T, group] (fp32 for MLS_FP32 inputs), in this workspace.
 */
size_t mls_workspace_size(const mls_problem* p);

/*
 * Forward (Eq. 2, Eq. 3, weighted sum over sub-models).
 *   H[m]      device, [T, d_m] in_dtype      hidden states of sub-model m (may be NULL when T = 0)
 *   W[m]      device, [V, d_m] in_dtype      LM head of sub-model m
 *   targets   device, int32 [T]; < 0 = ignored token
 *   loss      device, fp32 [1]               the scalar objective
 *   tok_loss  device, fp32 [M, T]            L_m per token (0 for ignored tokens)
 *   tok_diag  device, fp32 [3, M, T] or NULL CE_m, Ld_m and KL_m = Ld_m - H(q) per token
 *   argmax    device, int32 [M, T] or NULL   argmax_v z_m (lowest index on ties)
 *   stats     device, fp32 [2, M, T]         logsumexp(z_m) and logsumexp(z_m / tau);
 *                                            the backward needs them
 *   ws        device workspace, ws_bytes >= mls_workspace_size(p)
 */
int mls_head_loss_fwd(const mls_problem* p, const void* const* H, const void* const* W,
                      const int32_t* targets, float* loss, float* tok_loss, float* tok_diag,
                      int32_t* argmax, float* stats, void* ws, size_t ws_bytes,
                      mls_stream_t stream);

/*
 * Backward: gradients of grad_scale * loss.
 *   stats     device, fp32 [2, M, T] as written by mls_head_loss_fwd for the same inputs
 *   dH[m]     device, fp32 [T, d_m]    overwritten with d(loss)/dH_m
 *   dW[m]     device, fp32 [V, d_m]    overwritten with d(loss)/dW_m (zeros when T = 0
 *                                      or no token counts; H[m], dH[m] may be NULL when T = 0)
 * The teacher's parameters get only the gradient of w_t * mean CE_t: Eq. 2 stops
 * the gradient through q.  The logits are recomputed, never read from memory.
 */
int mls_head_loss_bwd(const mls_problem* p, const void* const* H, const void* const* W,
                      const int32_t* targets, const float* stats, float grad_scale,
                      float* const* dH, float* const* dW, void* ws, size_t ws_bytes,
                      mls_stream_t stream);

/*
 * Evaluation metrics between sub-models (Sec. 3.2.2: pairwise KL divergence
 * and top-1 next-token agreement across the suite; App. A plots
 * KL(p_student || p_teacher)).  Forward only, softmax at temperature 1; tau,
 * alpha, w and the teacher index of `p` are not used.
 *   targets    device, int32 [T] or NULL: tokens with a target outside [0, V)
 *              are left out of the means (NULL: every token counts)
 *   tok_kl     device, fp32 [M, M, T]: KL(p_i || p_j) per token (diagonal 0)
 *   argmax     device, int32 [M, T] or NULL
 *   pair_stats device, fp32 [2, M, M]: mean KL(p_i || p_j) and the fraction of
 *              tokens on which argmax z_i == argmax z_j
 *   ws         device workspace, ws_bytes >= mls_workspace_size(p)
 */
int mls_head_pairwise(const mls_problem* p, const void* const* H, const void* const* W,
                      const int32_t* targets, float* tok_kl, int32_t* argmax, float* pair_stats,
                      void* ws, size_t ws_bytes, mls_stream_t stream);

/*
 * Inter-model junction (Eq. 1) between sub-model m (width D_m = d_prev) and
 * sub-model m+1 (width D_{m+1} = d_next), per token:
 *   o~ = o * ||e||_2 / ||o||_2   (o~ = 0 when ||o|| = 0)
 *   x  = concat(o~, e)  if embed_first == 0  (the prose: the first D_m channels
 *                                             carry sub-model m)
 *   x  = concat(e, o~)  if embed_first != 0  (Eq. 1's written order)
 *   o  device [T, d_prev], e device [T, d_next - d_prev], x device [T, d_next],
 *   all row-major in in_dtype (MLS_BF16 or MLS_FP32), 16-byte aligned, rows a
 *   multiple of 16 bytes; sums are fp32.
 * Backward: g = dL/dx [T, d_next]; d_o [T, d_prev] and d_e [T, d_next - d_prev]
 * are overwritten (same storage type) with
 *   dL/do = s (g_o - o (g_o . o) / ||o||^2),  dL/de = g_e + s (g_o . o) e / ||e||^2,
 *   s = ||e|| / ||o||  (both terms 0 when ||o|| = 0).
 * Asynchronous on `stream`; returns 0 or a negative MLS_ERR_* code.
 */
int mls_junction_fwd(int64_t T, int32_t d_prev, int32_t d_next, int32_t in_dtype,
                     int32_t embed_first, const void* o, const void* e, void* x,
                     mls_stream_t stream);
int mls_junction_bwd(int64_t T, int32_t d_prev, int32_t d_next, int32_t in_dtype,
                     int32_t embed_first, const void* o, const void* e, const void* g,
                     void* d_o, void* d_e, mls_stream_t stream);

/*
 * Speculative-decoding verify step for a nested draft / verifier pair
 * (Sec. 2, "Speculative Decoding": sub-model m drafts gamma tokens, a larger
 * sub-model m' verifies them in one pass; Sec. 3.2.3 samples with temperature
 * 0.4 and nucleus p = 0.9, or greedily).  Standard speculative sampling over
 * B independent sequences; position i of sequence b is row b*gamma + i of
 * H_draft and row b*(gamma+1) + i of H_verify.
 *   q_i = nucleus(softmax(H_draft[i] W_draft^T / temperature))     i < gamma
 *   p_i = nucleus(softmax(H_verify[i] W_verify^T / temperature))   i <= gamma
 *   nucleus(r): tokens ordered by probability (descending, then by index) are
 *   kept through the first one at which the cumulative probability reaches
 *   top_p, then renormalised (top_p = 1 keeps every token).
 *   Drafted token x_i is accepted iff q_i(x_i) > 0 and u[b,i,0] q_i(x_i) < p_i(x_i);
 *   n_accepted[b] = k, the number accepted before the first rejection, and
 *   next_token[b] = sample(max(0, p_k - q_k), u[b,k,1]) (sample(p_k, u[b,k,1])
 *   when that residual is all zero), or sample(p_gamma, u[b,gamma,1]) when all
 *   gamma were accepted, with sample(r, u) = the smallest v such that
 *   sum_{w <= v} r_w > u * sum_w r_w.
 *   greedy != 0: x_i is accepted iff it is the argmax of the verifier's
 *   logits (lowest index on ties) and next_token is that argmax at position k;
 *   the draft model, temperature, top_p and uniforms are not used (H_draft,
 *   W_draft and uniforms may be NULL).
 * Arguments (device pointers unless stated):
 *   p            host; d_draft/d_verify: widths; in_dtype: storage of H and W
 *   H_draft      [B*gamma, d_draft], W_draft [V, d_draft]      (in_dtype)
 *   H_verify     [B*(gamma+1), d_verify], W_verify [V, d_verify]
 *   draft_tokens int32 [B, gamma]; a token outside [0, V) is rejected
 *   uniforms     fp32 [B, gamma+1, 2] in [0, 1): acceptance and sampling draws
 *   n_accepted   int32 [B] (written), next_token int32 [B] (written)
 *   ws           workspace of mls_spec_workspace_size(p) bytes, 256-byte aligned;
 *                when sampling it holds an fp32 row of unnormalised
 *                probabilities per verify position (greedy: per-tile maxima only).
 * Sampling supports V <= 4096 * 256 and gamma <= 1024 (MLS_ERR_UNSUPPORTED
 * beyond); greedy has neither limit.
 * Logits are fp32 sums of the stored-type products; probabilities are fp32, so a
 * decision that the exact values leave within rounding of a threshold may go
 * either way.  Asynchronous; returns 0 or a negative MLS_ERR_* code (nothing
 * launched).  B = 0 is a no-op.
 */
typedef struct {
  int32_t B;            /* sequences, >= 0 */
  int32_t gamma;        /* drafted tokens per sequence, >= 0 */
  int64_t V;            /* vocabulary, 1 .. 2^31 - 1 */
  int32_t d_draft;      /* width of the draft sub-model (unused when greedy) */
  int32_t d_verify;     /* width of the verifier sub-model */
  float temperature;    /* > 0 (paper: 0.4) */
  float top_p;          /* (0, 1] (paper: 0.9) */
  int32_t greedy;       /* non-zero: greedy verification */
  int32_t in_dtype;     /* MLS_BF16 or MLS_FP32 */
} mls_spec_problem;

size_t mls_spec_workspace_size(const mls_spec_problem* p);
int mls_spec_verify(const mls_spec_problem* p, const void* H_draft, const void* W_draft,
                    const void* H_verify, const void* W_verify, const int32_t* draft_tokens,
                    const float* uniforms, int32_t* n_accepted, int32_t* next_token, void* ws,
                    size_t ws_bytes, mls_stream_t stream);

/*
 * Synchronises `stream`, then returns the status bits (MLS_STATUS_*) recorded by
 * the device on the current device since the last call and clears them; returns
 * a negative MLS_ERR_CUDA if the synchronisation or the read failed.
 */
int mls_get_status(mls_stream_t stream);

/* Static description of a return code or status bit. */
const char* mls_strerror(int code);

/*
 * Forward without a caller-provided workspace (the paper has no counterpart;
 * this is an interface convenience).  Same operation, arguments and outputs as
 * mls_head_loss_fwd minus ws/ws_bytes: the scratch it needs (per-CTA partial
 * row states and per-block sums) lives in a fixed device array of
 * MLS_NOALLOC_SCRATCH_BYTES that the library reserves on every GPU that loads
 * it, for the life of the process.  It calls no cudaMalloc or cudaFree and no
 * allocating library routine.  It is meant for callers that cannot allocate
 * device memory at the point of the call: a host program or plugin that has no
 * allocator to hand out a workspace, or a steady-state loop that must not call
 * cudaMalloc, which can synchronise the device and carve memory out of a pool
 * another allocator already owns.
 *   - A problem whose forward needs more than MLS_NOALLOC_SCRATCH_BYTES of
 *     scratch is rejected with MLS_ERR_WORKSPACE before anything is launched.
 *     (The benchmark workloads need at most about 36 MiB; mls_workspace_size
 *     reports the larger forward+backward requirement, not this one.)
 *   - The first call on a device looks up the array's device address on that
 *     device (cudaGetSymbolAddress); make that first call before any stream
 *     capture.
 *   - All calls on a device share the one array and it keeps the previous
 *     call's contents.  Nothing in it needs to start at zero: each call writes
 *     every word it later reads.  Calls whose kernels overlap on the GPU (other
 *     streams, other host threads) race on the array and corrupt each other's
 *     results; serialise them.
 */
#define MLS_NOALLOC_SCRATCH_BYTES (64u << 20)
int mls_head_loss_fwd_noalloc(const mls_problem* p, const void* const* H, const void* const* W,
                              const int32_t* targets, float* loss, float* tok_loss,
                              float* tok_diag, int32_t* argmax, float* stats, mls_stream_t stream);

/*
 * Kernel timing (a tracing aid; not part of the paper's method).  While
 * enabled, every kernel the library launches is bracketed by two CUDA events
 * recorded on the launch stream.  mls_profile_read synchronises on the last
 * event, then fills up to `n` records (kernel name, launch count, summed
 * device time in ms), aggregated by kernel since the last enable/read, and
 * returns how many kernels it saw; the records are cleared.  Host-side state
 * only; thread-unsafe with concurrent calls on other threads.
 */
typedef struct {
  const char* name;   /* static string, e.g. "head_fwd" */
  int launches;
  double total_ms;
} mls_kernel_time;

int mls_profile_enable(int on);
int mls_profile_read(mls_kernel_time* out, int n);

#ifdef __cplusplus
}
#endif

#endif /* MLS_H */
