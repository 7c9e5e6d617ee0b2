/*
 * dvi.h -- C-ABI of the GB300 (sm_103a) DVI library.
 *
 * DVI (Draft, Verify & Improve, arxiv 2510.05421) splits one decoder at layer
 * k (Sec. 3.1): layers 1..k plus a LoRA drafter head greedily propose k_spec
 * tokens; the frozen layers k+1..L plus the LM head verify the whole block in
 * one multi-query pass; the longest agreeing prefix is committed and the KV
 * cache rolled back past it (Sec. 3.3); the logged accept/reject tuples drive
 * an online KL->RL update of the drafter head (Sec. 3.4).
 *
 * Conventions shared by every call
 *  - Memory.  The caller owns all device memory: weights, the workspace and
 *    every input/output buffer.  The library never allocates or frees device
 *    memory.  A context keeps raw pointers to the weights and the workspace;
 *    both must outlive it.
 *  - Asynchrony.  Every call only enqueues work on the context's stream and
 *    returns.  Argument errors are reported synchronously through the return
 *    value.  Errors found on the device (non-finite logits or loss, KV or
 *    buffer capacity, a bounded wait that ran out) set bits of a device
 *    status word that dvi_get_stats() reads.
 *  - Threads.  A context is used by one host thread at a time.  No C++
 *    exception crosses this interface.
 *  - Layout.  Matrices are row-major with the output feature as the row
 *    (torch nn.Linear layout): W[out][in].  Token ids are int32.
 */
#ifndef DVI_H_
#define DVI_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct dvi_ctx dvi_ctx;           /* opaque, host-side */
typedef struct CUstream_st* dvi_stream;   /* a cudaStream_t */

typedef enum {
  DVI_OK = 0,
  DVI_ERR_INVALID_ARG = -1,
  DVI_ERR_CAPACITY = -2,
  DVI_ERR_NONFINITE = -3,
  DVI_ERR_CUDA = -4,
  DVI_ERR_UNIMPLEMENTED = -5,
  DVI_ERR_TIMEOUT = -6
} dvi_status;

/* bits of dvi_stats.device_status */
enum {
  DVI_DEV_NONFINITE = 1,   /* a NaN/Inf logit, or a non-finite update loss (update skipped) */
  DVI_DEV_TIMEOUT = 2,     /* a bounded device wait gave up */
  DVI_DEV_KV_FULL = 4,     /* a KV row fell past max_seq_len (row not written) */
  DVI_DEV_BAD_TOKEN = 8,   /* a token id outside [0, vocab) */
  DVI_DEV_LOG_FULL = 16    /* the replay buffer was full; tuples of a step were dropped */
};

typedef enum { DVI_F32 = 0, DVI_BF16 = 1 } dvi_dtype;

/* The decoder (Sec. 3.1; the backbone is Llama-style: pre-norm RMSNorm,
 * RoPE rotate-half, SwiGLU, GQA).  dtype is the storage type of the weight
 * matrices and the KV cache.  The residual stream, norm gains, LoRA factors
 * and logits are float32; with bf16, the activations that meet a weight
 * matrix in a tensor-core product (and the queries and probabilities of the
 * attention) enter it as a bf16 pair hi + lo, so the products carry the
 * rounding of the stored weights and cache only. */
typedef struct {
  int n_layers;       /* L */
  int d_model;        /* d, a multiple of 128 */
  int n_heads;        /* H_q */
  int n_kv_heads;     /* H_kv, divides H_q */
  int head_dim;       /* 64 or 128 */
  int d_ffn;          /* F */
  int vocab;          /* V */
  int split_k;        /* k: draft path = layers 1..k, verify path = k+1..L; 1 <= k <= L */
  int lora_rank;      /* r of A_s [V][r], B_s [r][d]; 0 = no LoRA */
  float lora_gamma;   /* gamma_s */
  float rms_eps;      /* 1e-5 */
  float rope_theta;   /* 10000 */
  int dtype;          /* dvi_dtype */
} dvi_model_config;

typedef struct {
  int batch;            /* B sequences decoded together */
  int k_spec;           /* K: drafted tokens per step, 1 <= K <= 16 (K + bonus <= 16) */
  int max_seq_len;      /* KV rows per sequence: prompt + generated + K */
  int log_steps;        /* decode steps the replay buffer holds between updates (U) */
  int head_mode;        /* 0: train LoRA A_s, B_s on the frozen W^(S); 1: train W^(S) itself
                           (the LoRA factors, if any, stay frozen; the workspace then holds
                           the Adam moments of W^(S), an f32 master copy of it when dtype is
                           bf16, and the gradient buffer: 12 (f32) or 16 (bf16) B per entry) */
  int max_prefill_chunk;/* rows per prefill pass, a multiple of 16: bf16 16..4096 (0 = 1024),
                           f32 16..128 (0 = 128).  A bf16 pass runs its projections on the
                           prefill kernel (128 token rows x 256 features per tile), so the
                           weights stream from HBM about once per pass. */
  int use_graphs;       /* capture the decode step in a CUDA graph on first use */
  int bonus;            /* 0: verify the K drafted rows and commit min(m+1, K) tokens (Sec. 3.3
                           emits y*_{n+m+1}, which the K verify rows hold only for m < K);
                           1: one more shallow pass on t~_K and a (K+1)-th verify row, so the
                           correction y*_{n+K+1} exists at m = K and every step commits m+1
                           tokens.  K + bonus <= 16. */
  int persistent;       /* 0: one kernel per projection.  1: bf16 decode passes of up to 64
                           rows run each layer's O, gate/up and down projections and the next
                           layer's QKV as one persistent launch (attention stays a launch of
                           its own); the context then needs every CTA of that launch resident
                           at once (two per SM) and ignores the flag when they do not fit.
                           Results differ from mode 0 in summation order only. */
  int chain_counters;   /* 0: each launch of a decode pass waits for its predecessor's whole
                           grid (programmatic dependent launch).  1: bf16 decode passes
                           (draft, verify, AR step; not with persistent = 1) chain their
                           projection, attention and head launches through per-launch
                           completion counters: each CTA adds 1 with release semantics
                           after its last write and the next launch polls the count with
                           acquire semantics (bounded: DVI_DEV_TIMEOUT).  Same arithmetic,
                           bit-identical results. */
  int megakernel;       /* 0: the draft passes run one kernel per projection, attention and
                           head.  1: bf16 contexts of at most 2 sequences with k <= 16 draft
                           layers (GQA groups of 1, 2, 4 or 8 -- 8 at head_dim 64 only --,
                           head_dim 64 or 128, d a multiple of 128)
                           run the whole draft phase -- every draft pass's k layers, the
                           drafter head with its argmax, the hand-off of h_k to the verify
                           rows -- as one persistent launch of one CTA per SM (Sec. 3.3
                           draft rollout), and the greedy AR step runs its first k layers
                           the same way, so the DVI stream stays bit-identical to AR.  Its
                           projections are row-split GEMVs on f32 activations and its
                           attention runs on warp MMAs (online softmax per warp); its phases
                           meet at completion counters with bounded waits.  Ignored when the
                           shape or the device does not allow it (stats: megakernel_ctas). */
} dvi_runtime_config;

typedef struct {
  const void* attn_norm;   /* [d] f32 */
  const void* wq;          /* [H_q*hd][d] */
  const void* wk;          /* [H_kv*hd][d] */
  const void* wv;          /* [H_kv*hd][d] */
  const void* wo;          /* [d][H_q*hd] */
  const void* ffn_norm;    /* [d] f32 */
  const void* w_gate;      /* [F][d] */
  const void* w_up;        /* [F][d] */
  const void* w_down;      /* [d][F] */
} dvi_layer_weights;

/* Device pointers, caller-owned, read for the whole life of the context.
 * final_norm and lora_b must be 16-byte aligned (dvi_create returns
 * DVI_ERR_INVALID_ARG otherwise), and so must every bf16 weight matrix.
 * draft_head (W^(S)) may alias lm_head (W^(V)) only when head_mode == 0.
 * lora_a / lora_b are updated in place by dvi_update_drafter (head_mode 0);
 * draft_head is updated in place in head_mode 1: with dtype bf16 the
 * optimizer steps an f32 master copy (taken from draft_head by dvi_create)
 * and writes its bf16 rounding back to draft_head after every update. */
typedef struct {
  const void* embed;              /* [V][d] */
  const dvi_layer_weights* layers;/* host array of L entries */
  const void* final_norm;         /* [d] f32 */
  const void* lm_head;            /* W^(V) [V][d], frozen */
  void* draft_head;               /* W^(S) [V][d] */
  float* lora_a;                  /* A_s [V][r] f32 */
  float* lora_b;                  /* B_s [r][d] f32 */
} dvi_weights;

/* Drafter-update hyper-parameters (Sec. 3.4).  objective: 0 = the KL->RL
 * schedule (L_fast, plus L_policy once t >= t_warmup), 1 = KL only, 2 = PG
 * only (REINFORCE), 3 = reward-masked CE only (the ablations of Sec. 4.3).
 * optimizer: 0 = bias-corrected Adam, 1 = SGD. */
typedef struct {
  int objective;
  int optimizer;
  float lr, beta1, beta2, adam_eps;
  float tau;                                  /* KD temperature */
  float lambda0, lambda_kl_min, lambda_pg_max;
  int t_warmup, t_ramp;
  float w_ce, w_ent, w_rl_max;
  float beta0, beta_min, t_beta;              /* beta(t) of L_policy */
  float baseline_rho;                         /* EMA constant of the reward baseline b */
  int keep_grad_w;                            /* head_mode 1: also store dL/dW^(S) in DVI_BUF_GRAD_W
                                                 (4 more bytes of traffic per W^(S) entry) */
} dvi_update_config;

typedef struct {
  int64_t steps;          /* draft_verify_commit calls */
  int64_t drafted;        /* sum over sequences of K per step */
  int64_t accepted;       /* sum of m (mean accepted length = accepted / (steps * B)) */
  int64_t committed;      /* tokens committed by decode steps */
  int64_t updates;        /* drafter updates applied */
  int64_t kernel_launches;/* kernels this context enqueued (graph replays count their nodes) */
  float last_loss;        /* objective of the last update */
  float last_kl, last_pg, last_ce, last_ent, last_rl, last_kl1;
  float last_accept_rate; /* accepted / logged rows of the last update's buffer */
  float baseline_b;       /* EMA reward baseline after the last update */
  int update_t;           /* completed updates t (the schedule's clock) */
  int device_status;      /* DVI_DEV_* bits */
  int persistent_ctas;    /* grid of the persistent projection launch (runtime option
                             persistent = 1 in effect), else 0 */
  int megakernel_ctas;    /* grid of the draft-phase megakernel (runtime option megakernel = 1
                             in effect), else 0 */
} dvi_stats;

/* Bytes of device workspace a context needs (KV caches, residual streams,
 * replay buffer, optimizer state, scratch).  0 for an invalid config. */
size_t dvi_workspace_bytes(const dvi_model_config* cfg, const dvi_runtime_config* rt);

/* "Load split model" (Sec. 3.1): validate the config, keep the weight
 * pointers, carve `workspace` (>= dvi_workspace_bytes, 256-byte aligned,
 * contents arbitrary) and enqueue its initialisation on `stream`.  Builds
 * the TMA descriptors of every weight matrix. */
dvi_status dvi_create(const dvi_model_config* cfg, const dvi_runtime_config* rt,
                      const dvi_weights* weights, void* workspace,
                      size_t workspace_bytes, dvi_stream stream, dvi_ctx** out);

/* Reset sequence `seq` and run its prompt (device int32 [n_tokens]) through
 * all L layers, filling the KV cache; the greedy next token (the first
 * generated token, committed) becomes the pending token of the sequence and
 * is written to d_first_token (device int32 [1]) when non-null. */
dvi_status dvi_prefill(dvi_ctx* ctx, int seq, const int32_t* d_tokens, int n_tokens,
                       int32_t* d_first_token);

/* One DVI step for all B sequences (Sec. 3.3): K greedy draft passes through
 * layers 1..k and the drafter head, one verify pass of the K (K+1 with the
 * bonus row) rows through layers k+1..L and the LM head, accept length m,
 * commit and rollback, and (when logging is on) the replay-buffer tuples of
 * positions 1..min(m+1, K).  Outputs (device, may be null): d_out_ids
 * [B][K + bonus] committed ids (the first d_n_committed[b] entries of row b
 * are valid: min(m+1, K), or m+1 with the bonus row), d_n_accepted [B] = m. */
dvi_status dvi_draft_verify_commit(dvi_ctx* ctx, int32_t* d_out_ids,
                                   int32_t* d_n_committed, int32_t* d_n_accepted);

/* Replay-buffer logging on (1, the default) or off (0) for later steps. */
dvi_status dvi_log(dvi_ctx* ctx, int enable);

/* One drafter-head update on every tuple logged since the last update
 * (Sec. 3.4), then clear the buffer and advance t.  With the per-row logit
 * gradients G [N][V] of the loss, head_mode 0 steps A_s and B_s with
 * dA = gamma G^T (U B^T) and dB = gamma (G A)^T U; head_mode 1 steps W^(S)
 * with dW = G^T U.  A non-finite loss skips the parameter step and sets
 * DVI_DEV_NONFINITE.  DVI_ERR_UNIMPLEMENTED in head_mode 0 without LoRA
 * factors (nothing to train). */
dvi_status dvi_update_drafter(dvi_ctx* ctx, const dvi_update_config* ucfg);

/* Baseline: one greedy autoregressive step of the full model for every
 * sequence (the speedup denominator of Sec. 4.1); commits one token each.
 * d_out_ids: device int32 [B] or null. */
dvi_status dvi_ar_step(dvi_ctx* ctx, int32_t* d_out_ids);

/* Synchronise the context's stream and copy the counters to *out. */
dvi_status dvi_get_stats(dvi_ctx* ctx, dvi_stats* out);

/* Message of the last synchronous error on this context ("" if none). */
const char* dvi_last_error(const dvi_ctx* ctx);

/* Free the host-side context (never the caller's device memory). */
dvi_status dvi_destroy(dvi_ctx* ctx);

/* Inspection of internal device buffers for tests and tools: sets *dptr and
 * *bytes for buffer `which` (DVI_BUF_*).  The memory stays owned by the
 * workspace. */
enum {
  DVI_BUF_LENS = 0,        /* int32 [B] committed KV length n per sequence */
  DVI_BUF_PENDING = 1,     /* int32 [B] pending (last committed) token */
  DVI_BUF_DRAFT_IDS = 2,   /* int32 [B][K+1]: pending, t~_1..t~_K of the last step */
  DVI_BUF_LOG_U = 3,       /* logged head inputs u = RMSNorm_final(h_k): f32 [cap][d]; bf16
                              [2][cap][d], a hi plane then a lo plane, u = hi + lo */
  DVI_BUF_LOG_LOGITS = 4,  /* f32 [cap][V] logged verifier logits */
  DVI_BUF_LOG_META = 5,    /* int32 [cap][6]: valid, a, r, i, prev_id, y* */
  DVI_BUF_GRAD_A = 6,      /* f32 [V][r] last dL/dA */
  DVI_BUF_GRAD_B = 7,      /* f32 [r][d] last dL/dB */
  DVI_BUF_X_DRAFT = 8,     /* f32 [B][d] residual stream of the draft pass */
  DVI_BUF_X_VERIFY = 9,    /* f32 [B*K][d] h_k rows, then h_L after verify */
  DVI_BUF_K_CACHE = 10,    /* dtype [L][B][H_kv][max_seq_len][hd] */
  DVI_BUF_V_CACHE = 11,
  DVI_BUF_STATUS = 12,     /* int32 device status word */
  DVI_BUF_GRAD_W = 13,     /* f32 [V][d] last dL/dW^(S) (head_mode 1, written when keep_grad_w) */
  DVI_BUF_Z = 14,          /* f32 [cap][V] drafter logits z of the buffer rows: logged by the drafter
                              head while drafting (head_mode 0; A, B and W^(S) change only at an
                              update, which empties the buffer), else recomputed by the update */
  DVI_BUF_COUNT
};
dvi_status dvi_debug_buffer(dvi_ctx* ctx, int which, void** dptr, size_t* bytes);

/* Device timing of the phases for measurement: while enabled, CUDA events
 * are recorded on the context's stream around the draft phase (0), the
 * verify phase (1) and the drafter update (2) of every call. */
dvi_status dvi_timing(dvi_ctx* ctx, int enable);

/* Synchronise the stream, then return per phase the summed milliseconds
 * ms[3] and the number of timed calls counts[3] since the last read. */
dvi_status dvi_get_timing(dvi_ctx* ctx, double* ms, int* counts);

/* Y[M][n_out] = X[M][K] . W[n_out][K]^T through the library's projection
 * kernel (tcgen05 for bf16, FP32 FMA for f32), with X float32 (for bf16
 * weights carried as a bf16 pair hi + lo, about 16 significant bits) and Y
 * float32, on the context's stream.  M <= 256.
 * A building block exposed for tests of the projection kernel itself. */
dvi_status dvi_linear(dvi_ctx* ctx, const void* d_w, int n_out, int k_in,
                      const float* d_x, int m_rows, float* d_y);

/* Y[M][n_out] = X[M][K] . W[n_out][K]^T like dvi_linear, for callers that
 * cannot allocate device memory (code inside another framework's memory
 * pool or a fixed device-memory budget, plug-ins that are handed only their
 * input and output buffers).  It needs no context and allocates nothing:
 * the split-K scratch is a fixed array inside the library, 8 MiB of partial
 * sums plus 4096 tile counters, which every GPU that loads the library
 * holds until the process exits.  The paper has no counterpart to this
 * call; it is a deployment convenience.
 *  - dtype: DVI_BF16 (tcgen05 path; k_in % 8 == 0, 16-byte aligned d_w and
 *    d_x) or DVI_F32 (FP32 FMA path).  d_w [n_out][k_in] in that dtype,
 *    d_x [m_rows][k_in] f32, d_y [m_rows][n_out] f32, all device pointers
 *    owned by the caller, on the current device; 1 <= m_rows <= 256.  With
 *    bf16 weights the kernel carries each f32 input as a bf16 pair hi + lo
 *    (about 16 significant bits), so only the weights are rounded.
 *  - Every device of the process has its own scratch and its own kernel
 *    attributes, each set up on the first call with that device current.
 *  - Shapes whose split plan needs more scratch than the fixed array holds
 *    return DVI_ERR_CAPACITY (with a message on stderr); for example a
 *    4096 x 4096 weight fits for up to 32 rows.
 *  - The first call on a device looks up the scratch address for that
 *    device; make that first call before any stream capture.
 *  - All calls on a device share the one scratch array, and it keeps the
 *    last call's contents (the counters are cleared at the start of each
 *    call): calls that overlap on the GPU, e.g. on two streams, race. */
dvi_status dvi_linear_noalloc(int dtype, const void* d_w, int n_out, int k_in, const float* d_x,
                              int m_rows, float* d_y, dvi_stream stream);

#ifdef __cplusplus
}
#endif
#endif /* DVI_H_ */
