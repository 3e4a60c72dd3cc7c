/*
 * cora.h -- C ABI of the GB300 (sm_103a) CORA-Diff decoding library.
 *
 * CORA-Diff (Confidence-Oriented Residual Acceptance) keeps a frozen
 * diffusion language model and its dense bidirectional forward at every
 * executed step, then (Sec. 3):
 *   Eq. 1  takes the top-1 prediction and confidence of every active position,
 *          x_hat_i = argmax_v p_iv, c_i = max_v p_iv, p = softmax(logits);
 *          the original low-confidence transfer rule fixes the k highest-
 *          confidence unresolved positions of the active block (Sec. 3.1);
 *   Eq. 2  counts, per unresolved position, how many consecutive executed
 *          steps kept the same top-1 prediction (0 at its first step);
 *   Eq. 3  accepts a residual position (one the transfer rule left
 *          unresolved) when c_i >= delta_p and m_i >= m;
 *   Eq. 4  writes accepted tokens into the canvas (they stay visible as
 *          context) and removes both sets from the unresolved set;
 *   and ends the block, skipping its remaining dense passes, once no
 *   position of the block is unresolved (Sec. 3 overview; Sec. 3.3).
 * In this header delta_p is called `tau` and the persistence window m is `K`.
 *
 * Conventions
 *  - Every call returns an int status: CORA_OK (0) or a negative error code.
 *    cora_last_error() returns a message for the calling thread's last error.
 *    Arguments are validated before any launch; nothing is launched on error.
 *  - "device" pointers are CUDA device (or managed) memory of the current
 *    device; "host" pointers are ordinary host memory; "any" pointers may be
 *    either (they are read with cudaMemcpyDefault).
 *  - Caller-owned buffers are borrowed for the duration of the call only.
 *    Objects returned through `**out` are owned by the library and released
 *    with their destroy call.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *    stream).  Calls taking a stream are asynchronous unless stated.
 *  - bf16 tensors are passed as uint16_t bit patterns; matrices are row-major.
 *  - No exception crosses this boundary; the library never falls back to a
 *    CPU implementation.
 */
#ifndef CORA_H_
#define CORA_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define CORA_API __attribute__((visibility("default")))
#else
#define CORA_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

#define CORA_OK 0
#define CORA_EINVAL -1   /* bad argument: shape, pointer, range */
#define CORA_ECUDA -2    /* a CUDA runtime/driver call failed */
#define CORA_ENOMEM -3   /* device allocation failed */
#define CORA_ETIMEOUT -4 /* a kernel's bounded wait expired; the error word was set */
#define CORA_ESTATE -5   /* call not valid in the object's current state */

/* Position states of the generation canvas. */
#define CORA_UNRESOLVED 0  /* still masked: in U^(s) */
#define CORA_TRANSFERRED 1 /* fixed by the original transfer rule: in T^(s) */
#define CORA_ACCEPTED 2    /* accepted by the residual gate: in A^(s) */
#define CORA_EOS_FILLED 3  /* set to the EOS id after a block that committed it (EOS-aware stop) */

/* Returns the message of the calling thread's last failed call ("" if none). */
CORA_API const char* cora_last_error(void);

/* Library ABI version (major * 100 + minor). */
CORA_API int cora_version(void);

/* ---------------------------------------------------------------------------
 * Backbone description.  A pre-norm bidirectional Transformer: token
 * embedding; per layer RMSNorm -> fused QKV projection -> RoPE (rotate-half
 * pairs (j, j + head_dim/2), angle pos * rope_theta^(-2j/head_dim)) ->
 * non-causal softmax attention with n_kv_heads groups -> output projection +
 * residual -> RMSNorm -> SwiGLU FFN (silu(x W_gate^T) * (x W_up^T)) W_down^T +
 * residual; final RMSNorm and an untied LM head.  This is the frozen dense
 * pass the paper runs unchanged at every executed step (Sec. 3, Sec. 4.1).
 * Constraints: d_model % 128 == 0, head_dim in {64, 128},
 * n_heads % n_kv_heads == 0, (n_heads * head_dim) % 64 == 0,
 * ((n_heads + 2 * n_kv_heads) * head_dim) % 128 == 0, vocab >= 2,
 * 0 <= mask_id < vocab.
 * ------------------------------------------------------------------------- */
typedef struct cora_model_config {
  int32_t n_layers;
  int32_t d_model;
  int32_t n_heads;
  int32_t n_kv_heads;
  int32_t head_dim;
  int32_t ffn;
  int32_t vocab;
  int32_t mask_id;
  float rope_theta;
  float norm_eps;
} cora_model_config;

/* Weights in nn.Linear layout ([out_features, in_features], row-major),
 * "any" pointers, every tensor of the element type `dtype` names:
 *   CORA_DTYPE_BF16  bf16 bit patterns (uint16_t), copied as they are;
 *   CORA_DTYPE_F32   IEEE float32, converted on the device to bf16 (round to
 *                    nearest, ties to even), the precision the kernels
 *                    compute in (the paper's backbones run in bf16, Sec. 4.1).
 * Per-layer members point to host arrays of n_layers tensor pointers.  Norm
 * weights may be NULL (all ones).
 *   embed    [vocab, d]           lm_head [vocab, d]        final_norm [d]
 *   wq [n_heads*hd, d]  wk, wv [n_kv_heads*hd, d]  wo [d, n_heads*hd]
 *   w_gate, w_up [ffn, d]         w_down [d, ffn]     attn_norm, ffn_norm [d]
 * The library copies them into its own device layout (fused QKV, gate/up
 * interleaved in 128-row groups, ffn padded to a multiple of 128 with zeros);
 * float32 host tensors pass through a device staging buffer of at most
 * 256 MiB.  The caller may free its copies when cora_model_create returns.
 * A zero-initialised struct means bf16 (dtype 0). */
#define CORA_DTYPE_BF16 0
#define CORA_DTYPE_F32 1
typedef struct cora_weights {
  const void* embed;
  const void* lm_head;
  const void* final_norm;
  const void* const* attn_norm;
  const void* const* wq;
  const void* const* wk;
  const void* const* wv;
  const void* const* wo;
  const void* const* ffn_norm;
  const void* const* w_gate;
  const void* const* w_up;
  const void* const* w_down;
  int32_t dtype; /* CORA_DTYPE_* */
} cora_weights;

typedef struct cora_model cora_model;
typedef struct cora_session cora_session;

/* Creates a device-resident model on the current device (synchronous).
 * Errors: CORA_EINVAL (config constraint, NULL tensor, unknown dtype),
 * CORA_ENOMEM, CORA_ECUDA. */
CORA_API int cora_model_create(const cora_model_config* cfg, const cora_weights* w, cora_model** out);
CORA_API int cora_model_destroy(cora_model* m);

/* ---------------------------------------------------------------------------
 * Decoding session: a batch of B independent sequences, each a canvas of
 * prompt_len prompt ids followed by gen_len positions initialised to mask_id
 * (Sec. 3.1), decoded in blocks of block_len positions with a horizon of
 * steps_per_block executed steps per block.  Each sequence keeps its own
 * block index, step index and pass count; a batched step runs while any
 * sequence is unfinished (rows of finished sequences are computed and
 * ignored).  Persistence counters reset at the start of every block.
 *   prompt   "any" int32 [B, prompt_len], ids in [0, vocab)
 *   tau      confidence threshold delta_p of Eq. 3 (compared in fp32; tau > 1
 *            switches the gate off)
 *   K        persistence window m of Eq. 3; K < 0 means infinity (gate off)
 * Constraints: B >= 1, prompt_len >= 0, gen_len % block_len == 0,
 * 1 <= block_len <= 32, steps_per_block >= 1, B * block_len <= 256.
 * Synchronous.  Errors: CORA_EINVAL, CORA_ENOMEM, CORA_ECUDA. */
CORA_API int cora_session_create(cora_model* m, int32_t batch, const int32_t* prompt, int32_t prompt_len, int32_t gen_len,
                        int32_t block_len, int32_t steps_per_block, float tau, int32_t K, cora_session** out);
CORA_API int cora_session_destroy(cora_session* s);

/* Decoding variants: the ablations the paper discusses around Sec. 3 (its
 * transfer schedule, where persistence starts counting, an EOS-aware stop).
 * All-zero options but eos_id = -1 are the method as described, which is
 * what cora_session_create uses.  Prefix-cache sessions run cora_session_run
 * as a host loop (one graph per block). */
#define CORA_SCHEDULE_FIXED 0      /* k_s from the block length: floor(BL/T), the first BL mod T steps +1 */
#define CORA_SCHEDULE_REMAINING 1  /* k_s = ceil(|U| / (T - s)), |U| = unresolved positions of the block */
#define CORA_PERSIST_BLOCK 0       /* Eq. 2 counters start at each block's first pass */
#define CORA_PERSIST_CARRY 1       /* counters from a position's first executed pass: every pass runs Eq. 1
                                      on every generation row (LM head over B * gen_len rows, in chunks of
                                      256) and updates Eq. 2 for every unresolved position */
#define CORA_CACHE_NONE 0          /* the dense pass at every executed step (Sec. 3) */
#define CORA_CACHE_PREFIX 1        /* a block's first pass is dense and keeps every layer's keys/values; its
                                      later passes recompute only the rows from the active block to the end
                                      of the canvas, attending to the kept keys/values of earlier positions.
                                      The sequences of a batch then move to the next block together (a
                                      sequence whose block ended waits; its own passes and tokens are those
                                      of a batch of one).  Not combined with CORA_PERSIST_CARRY;
                                      needs block_len == 32. */
typedef struct cora_decode_options {
  int32_t schedule;     /* CORA_SCHEDULE_* */
  int32_t persistence;  /* CORA_PERSIST_* */
  int32_t eos_id;       /* -1: none.  Else the EOS-aware stop: once a block terminates holding this id, the
                           sequence finishes and every later generation position takes the id
                           (state CORA_EOS_FILLED); later blocks execute no pass.  Must be a
                           vocabulary id other than the mask id. */
  int32_t cache;        /* CORA_CACHE_* */
} cora_decode_options;

/* cora_session_create with decoding options (NULL = defaults).  The options
 * are fixed for the session's lifetime (they are baked into its graphs).
 * Errors as cora_session_create; CORA_EINVAL for an unknown or unsupported
 * option value. */
CORA_API int cora_session_create_ex(cora_model* m, int32_t batch, const int32_t* prompt, int32_t prompt_len,
                                    int32_t gen_len, int32_t block_len, int32_t steps_per_block, float tau,
                                    int32_t K, const cora_decode_options* opt, cora_session** out);

/* Re-initialises the canvas from a new prompt (same shapes) and resets every
 * block/step/pass counter.  `prompt` is "any".  Synchronous. */
CORA_API int cora_session_reset(cora_session* s, const int32_t* prompt);

/* One executed denoising step (Sec. 3.1: step s of block b of the fixed
 * horizon) for every unfinished sequence, at that sequence's own (block,
 * step): dense forward over the whole canvas, final RMSNorm and LM head on the
 * active block's rows only, Eq. 1 reduced on the fly (logits never stored),
 * then the transfer rule, Eq. 2-4 and block termination.  Runs as one CUDA
 * graph on the session's stream and waits for it.
 *   block, step  the (block, step) the caller expects every unfinished
 *                sequence to be at (0-based); -1 skips that check.  A
 *                sequence at another block or step fails the call with
 *                CORA_ESTATE before anything is launched (with B > 1 the
 *                sequences may drift apart: pass -1 then).
 *   conf_out     "any" float [B, block_len] or NULL (out): this step's c_i
 *                (Eq. 1) of the rows of each sequence's active block
 *   argmax_out   "any" int32 [B, block_len] or NULL (out): this step's x_hat_i
 *                (Eq. 1), lowest id on ties
 *                (CORA_PERSIST_CARRY sessions: both are [B, gen_len], one
 *                entry per generation position)
 *   done_out     "any" uint8 [B] or NULL (out): 1 when sequence b's block has
 *                no unresolved position after this step (the block ended and
 *                its remaining dense passes are skipped), or the sequence had
 *                already finished; 0 otherwise
 * Rows of a sequence that had finished before the step hold values computed
 * and ignored.  Errors: CORA_ESTATE (already finished, or block/step differ),
 * CORA_ETIMEOUT, CORA_ECUDA. */
CORA_API int cora_denoise_step(cora_session* s, int32_t block, int32_t step, float* conf_out, int32_t* argmax_out,
                               uint8_t* done_out);

/* Host-side flag, no device work: *finished_out = 1 once every sequence of
 * the session has finished all its blocks (as of the last completed call). */
CORA_API int cora_session_finished(cora_session* s, uint8_t* finished_out);

/* Runs cora_denoise_step until every sequence has finished (the decode loop
 * of Sec. 3, Fig. 2), as ONE graph launch: a conditional WHILE node around
 * the step, whose condition a device kernel sets after each step's gate (all
 * sequences finished, an error, or n_blocks * T steps end it), so no host
 * round trip separates the passes.  Where the runtime cannot build that
 * graph, the same loop runs on the host, one cora_denoise_step at a time.
 *   steps_out      host int32 or NULL (out): batched steps executed by this call
 *   on_device_out  host uint8 or NULL (out): 1 when the device loop ran
 * Synchronous.  Errors: CORA_ESTATE (already finished, or unfinished after
 * the horizon), CORA_ETIMEOUT, CORA_ECUDA. */
CORA_API int cora_session_run(cora_session* s, int32_t* steps_out, uint8_t* on_device_out);

/* Copies session state to host buffers (any pointer may be NULL; synchronous):
 *   tokens  int32 [B, prompt_len + gen_len]   canvas
 *   state   uint8 [B, gen_len]               CORA_UNRESOLVED/TRANSFERRED/ACCEPTED/EOS_FILLED
 *   persist int32 [B, block_len]             Eq. 2 counters of the active block
 *   prev    int32 [B, block_len]             previous executed step's x_hat (-1: none)
 *           (CORA_PERSIST_CARRY sessions: persist, prev, conf and argmax are
 *           [B, gen_len], one entry per generation position)
 *   ctrl    int32 [B, 4]                     {block, step, passes executed, finished}
 *   conf    float [B, block_len]             last step's c_i (Eq. 1)
 *   argmax  int32 [B, block_len]             last step's x_hat_i (Eq. 1)
 *   unmask  uint8 [B, block_len]             last step's T^(s) indicator
 *   accept  uint8 [B, block_len]             last step's A^(s) indicator */
CORA_API int cora_session_read(cora_session* s, int32_t* tokens, uint8_t* state, int32_t* persist, int32_t* prev,
                      int32_t* ctrl, float* conf, int32_t* argmax, uint8_t* unmask, uint8_t* accept);

/* Overwrites session state from host buffers (same layouts as
 * cora_session_read; NULL leaves a part unchanged).  Lets a caller resume a
 * decode at block/step granularity.  In a prefix-cache session, writing ctrl
 * at a block's step 0 (or at another block than the current one) makes the
 * next pass that block's dense first pass; a later step of the current block
 * keeps the keys/values its first pass kept.  Synchronous. */
CORA_API int cora_session_write(cora_session* s, const int32_t* tokens, const uint8_t* state, const int32_t* persist,
                       const int32_t* prev, const int32_t* ctrl);

/* Disagreement with the dense endpoint (Sec. 4): compares the generation
 * canvas of session s (a CORA decode) with that of session `dense` (the same
 * model, prompts and shapes decoded with the gate off, i.e. Y*), after both
 * have run.  Per sequence b, host int64 [B] (out):
 *   n_acc       positions accepted by the residual gate (state CORA_ACCEPTED)
 *   n_acc_diff  of those, positions whose token differs from Y*
 *   n_out_diff  generation positions whose token differs from Y*
 * so that L^acc = n_acc_diff / max(1, n_acc) and L^out = n_out_diff / gen_len.
 * Synchronous.  Errors: CORA_EINVAL (NULL, shapes differ), CORA_ECUDA. */
CORA_API int cora_session_disagreement(cora_session* s, cora_session* dense, int64_t* n_acc, int64_t* n_acc_diff,
                                       int64_t* n_out_diff);

/* Launch classes reported by cora_session_profile_step. */
#define CORA_KIND_EMBED 0
#define CORA_KIND_RMSNORM 1
#define CORA_KIND_GEMM_QKV 2       /* QKV projection + RoPE epilogue */
#define CORA_KIND_ATTENTION 3
#define CORA_KIND_GEMM_O 4         /* output projection + residual */
#define CORA_KIND_GEMM_GATE_UP 5   /* gate/up projection + SwiGLU epilogue */
#define CORA_KIND_GEMM_DOWN 6      /* down projection + residual */
#define CORA_KIND_FINAL_NORM 7
#define CORA_KIND_LM_HEAD 8        /* fused LM head + Eq. 1 partials */
#define CORA_KIND_GATE 9           /* Eq. 1 combine + transfer rule + Eq. 2-4 */

/* Runs one cora_denoise_step without the CUDA graph, with CUDA events around
 * every kernel launch, for profiling.  It is a real step (state advances) and
 * runs the pass the next cora_denoise_step would run (in a prefix-cache
 * session: the block's dense first pass, or a pass over the rows from the
 * active block on).
 *   capacity  size of kinds/ms (>= 4 + 7 * n_layers)
 *   kinds     host int32 [capacity] (out): CORA_KIND_* of each launch, in order
 *   ms        host float [capacity] (out): device time of each launch
 *   n_out     host int32 (out): launches recorded
 * Synchronous. */
CORA_API int cora_session_profile_step(cora_session* s, int32_t capacity, int32_t* kinds, float* ms, int32_t* n_out);

/* The cudaStream_t (as void*) on which the session launches its work; a
 * caller may record events on it to time steps on the device. */
CORA_API int cora_session_stream(cora_session* s, void** out);

/* Number of batched steps (dense passes over the batch) executed since the
 * last reset. */
CORA_API int cora_session_batched_passes(cora_session* s, int64_t* out);

/* Full decode (Sec. 3, Fig. 2): creates or reuses the model's cached session
 * for these shapes, runs the decode with cora_session_run, and copies the
 * result to host memory.
 *   prompt      "any" int32 [B, P]
 *   tokens_out  host int32 [B, gen_len]   generated ids
 *   passes_out  host int64 [B]            executed dense passes per sequence
 *               (the paper's executed-step count; rho = passes / (blocks*T))
 *   batched_passes_out  host int64 [1] or NULL: batched steps executed
 * Synchronous.  Errors as cora_session_create / cora_denoise_step. */
CORA_API int cora_generate(cora_model* m, const int32_t* prompt, int32_t B, int32_t P, int32_t gen_len, int32_t block_len,
                  int32_t steps_per_block, float tau, int32_t K, int32_t* tokens_out, int64_t* passes_out,
                  int64_t* batched_passes_out);

/* cora_generate with decoding options (NULL = defaults; see
 * cora_session_create_ex). */
CORA_API int cora_generate_ex(cora_model* m, const int32_t* prompt, int32_t B, int32_t P, int32_t gen_len,
                              int32_t block_len, int32_t steps_per_block, float tau, int32_t K,
                              const cora_decode_options* opt, int32_t* tokens_out, int64_t* passes_out,
                              int64_t* batched_passes_out);

/* ---------------------------------------------------------------------------
 * Gate and transfer rule on device buffers (Eq. 2, transfer rule, Eq. 3,
 * Eq. 4) for B independent blocks of R positions (one warp per block):
 *   conf    device float [B, R]   c_i (Eq. 1)              (in)
 *   argmax  device int32 [B, R]   x_hat_i (Eq. 1)          (in)
 *   prev    device int32 [B, R]   previous x_hat, -1 none  (in/out)
 *   persist device int32 [B, R]   m_i (Eq. 2)              (in/out)
 *   state   device uint8 [B, R]   CORA_* position state    (in/out)
 *   tokens  device int32 [B, R]   canvas ids of the block  (in/out)
 *   k       transfer count of this step: the min(k, |U|) unresolved
 *           positions of highest confidence (ties: lower position) are fixed
 *   tau, K  Eq. 3 thresholds (fp32 compare; K < 0 = infinity)
 *   unmask, accept  device uint8 [B, R] (out): T^(s), A^(s) indicators
 *   done    device uint8 [B] (out): 1 when no position of the block is unresolved
 * Bit-exact with the paper's rule on identical inputs.  1 <= R <= 32.
 * Errors: CORA_EINVAL (shape, NULL), CORA_ECUDA (launch). */
CORA_API int cora_gate_transfer(const float* conf, const int32_t* argmax, int32_t* prev, int32_t* persist, uint8_t* state,
                       int32_t* tokens, int32_t B, int32_t R, int32_t k, float tau, int32_t K, uint8_t* unmask,
                       uint8_t* accept, uint8_t* done, void* stream);

/* Eq. 1 from materialised logits: device bf16 logits [rows, V] ->
 * conf (device float [rows]) and argmax (device int32 [rows], lowest id on
 * ties).  V >= 1.  Streams the logits once from HBM. */
CORA_API int cora_reduce_top1(const uint16_t* logits, int32_t rows, int32_t V, float* conf, int32_t* argmax, void* stream);

/* cora_reduce_top1 without any device allocation.  The paper has no
 * counterpart; this serves callers that must not allocate device memory when
 * they call it: applications whose memory pool already holds all device
 * memory (a cudaMalloc would fail or evict their cache), and latency-critical
 * loops that must stay out of the allocator (cudaMalloc and cudaFree
 * synchronise the device).
 * Scratch is a fixed array compiled into the library (832 KiB: 65536 partial
 * states + 16384 counters).  Same arguments, layout and results as
 * cora_reduce_top1; rows <= 16384, else CORA_EINVAL.
 * The array occupies device memory from the first use on a device of the
 * library part that holds it (with CUDA's default lazy module loading: the
 * first call of this function, or an earlier gate or Eq. 1 reduction call)
 * until the process exits; later calls reserve nothing.  So make one call
 * before a memory pool takes the whole device, and before any stream
 * capture: that first call on a device (with that device current) also looks
 * up the array's device address, which is then kept per device and looked up
 * again only when the current context changes (e.g. after cudaDeviceReset).
 * Calls share the array, so calls that may overlap on the GPU (different
 * streams without ordering) race; serialise them.  Each call clears the
 * counters it uses with cudaMemsetAsync on `stream` before its kernel. */
CORA_API int cora_reduce_top1_noalloc(const uint16_t* logits, int32_t rows, int32_t V, float* conf, int32_t* argmax,
                                      void* stream);

/* cora_reduce_top1 on [B, R, V] logits followed by cora_gate_transfer on the
 * result (the gate-isolation workload).  conf/argmax outputs are device
 * [B, R] and also serve as the gate's inputs. */
CORA_API int cora_reduce_gate(const uint16_t* logits, int32_t B, int32_t R, int32_t V, float* conf, int32_t* argmax,
                     int32_t* prev, int32_t* persist, uint8_t* state, int32_t* tokens, int32_t k, float tau,
                     int32_t K, uint8_t* unmask, uint8_t* accept, uint8_t* done, void* stream);

/* ---------------------------------------------------------------------------
 * Individual kernels of the dense pass, exposed for testing and profiling.
 * All pointers are device pointers.
 * ------------------------------------------------------------------------- */

/* Epilogues of cora_op_gemm. */
#define CORA_EPI_STORE_BF16 0 /* C = bf16(A B^T)                                    */
#define CORA_EPI_RESID_F32 1  /* H += A B^T (fp32 residual stream, H is C)          */
#define CORA_EPI_SWIGLU 2     /* C[:, 128t + j] = bf16(silu(acc[256t + j]) * acc[256t + 128 + j]) */
#define CORA_EPI_ROPE_BF16 3  /* C = bf16(rope(A B^T)) on columns < rope_cols, rows at position row % seq */

/* GEMM on tcgen05 tensor cores: acc = A[M, K] * B[N, K]^T with bf16 inputs
 * and fp32 accumulation (TMEM), TMA-fed, persistent over 128 x BN tiles.
 *   A     bf16 [M, K] row-major      B  bf16 [N, K] row-major (nn.Linear weight)
 *   C     bf16 [M, ldc] (STORE, ROPE, SWIGLU) or fp32 [M, ldc] (RESID)
 *   rope  fp32 [seq, head_dim/2, 2] (cos, sin) table for ROPE, else NULL
 * Constraints: K % 64 == 0, N % 128 == 0 (SWIGLU: N % 256 == 0), M >= 1,
 * pointers 16-byte aligned, row strides multiples of 16 bytes.
 * With ROPE the call also enqueues a transposed copy of the table into
 * stream-ordered memory (cudaMallocAsync on `stream`, freed after the GEMM):
 * the tile epilogue reads it frequency-major. */
CORA_API int cora_op_gemm(const uint16_t* A, const uint16_t* B, void* C, int32_t M, int32_t N, int32_t K, int32_t ldc,
                 int32_t epilogue, const float* rope, int32_t seq, int32_t head_dim, int32_t rope_cols,
                 void* stream);

/* How cora_op_gemm (and the dense pass) divides an M x N x K GEMM with the
 * given epilogue among CTAs on a GPU with num_sms SMs, computed on the host
 * with the same rules and the same segment walk the kernels use; no device
 * work, no CUDA call (usable without a GPU).  A test aid for the work split;
 * the paper has no counterpart.
 *   info  int32 [7], written: kernel (0 few-row, 1 one CTA per 128-row tile,
 *         2 CTA pairs on 256-row tiles), units (CTAs or CTA pairs), tiles,
 *         k-blocks per tile (K / 64), k-pieces per split tile (0: stream-K or
 *         whole tiles), 1 when two pieces share the fix-up, data-parallel waves
 *   seg   int32 [cap][6], written up to cap rows: unit, tile, first k-block,
 *         end k-block, row block, column block, in each unit's visiting order
 *         (kernel 0 has no segments)
 *   n_seg int32 [1], written: the number of segments (may exceed cap)
 * Errors: CORA_EINVAL for NULL pointers, M < 1, num_sms < 2, K % 64 != 0,
 * N % 128 != 0 or cap < 0. */
CORA_API int cora_gemm_plan(int32_t M, int32_t N, int32_t K, int32_t epilogue, int32_t num_sms, int32_t* info,
                            int32_t* seg, int32_t cap, int32_t* n_seg);

/* Non-causal attention of B sequences of length S from a fused QKV buffer
 * qkv bf16 [B*S, (Hq + 2*Hkv)*hd] (Q heads, then K heads, then V heads;
 * RoPE already applied) into out bf16 [B*S, Hq*hd]; softmax(QK^T/sqrt(hd))V,
 * query head h reading KV head h / (Hq/Hkv). */
CORA_API int cora_op_attention(const uint16_t* qkv, uint16_t* out, int32_t B, int32_t S, int32_t Hq, int32_t Hkv,
                      int32_t hd, void* stream);

/* cora_op_attention for the queries q_start .. q_start + q_len - 1 of every
 * sequence, against all S keys (the rows a prefix-cache pass recomputes;
 * Sec. 5 composes the method with cache reuse): qkv as above, bf16
 * [B*S, (Hq + 2*Hkv)*hd]; out bf16 [B*q_len, Hq*hd], q_len rows per
 * sequence.  0 <= q_start, 1 <= q_len, q_start + q_len <= S. */
CORA_API int cora_op_attention_rows(const uint16_t* qkv, uint16_t* out, int32_t B, int32_t S, int32_t Hq, int32_t Hkv,
                                    int32_t hd, int32_t q_start, int32_t q_len, void* stream);

/* RMSNorm rows: out bf16 [M, d] = x / sqrt(mean(x^2) + eps) * w, x fp32 [M, d],
 * w bf16 [d] (NULL = ones). */
CORA_API int cora_op_rmsnorm(const float* x, const uint16_t* w, uint16_t* out, int32_t M, int32_t d, float eps,
                    void* stream);

/* Fused LM head and Eq. 1: x bf16 [R, d] (already normalised), W bf16 [V, d]
 * -> conf float [R], argmax int32 [R]; logits are reduced in the GEMM
 * epilogue and never written to memory.  1 <= R <= 256, d % 64 == 0. */
CORA_API int cora_op_lm_head_top1(const uint16_t* x, const uint16_t* W, int32_t R, int32_t V, int32_t d, float* conf,
                         int32_t* argmax, void* stream);

/* ---------------------------------------------------------------------------
 * Seeded synthetic data (not part of the method): writes `count` bf16
 * approximate-normal samples, element i being output (start + i) of the
 * SplitMix64 stream `key`, Irwin-Hall(4) of its 16-bit fields scaled by
 * `scale` (fp32) and rounded to bf16.  Same bits as the Python generator. */
CORA_API int cora_synth_normal_bf16(uint16_t* out, int64_t count, uint64_t key, int64_t start, float scale, void* stream);

/* Reads (and with clear != 0, resets) the library's device error word for
 * the current device: 0 when no kernel has recorded a fault. */
CORA_API int cora_device_error(int32_t* code, int32_t clear);

/* Failure-detection self-check (every wait in the kernels is bounded, and an
 * expired wait is reported, not fatal).  Launches one CTA on the current device
 * whose thread waits, with the kernels' own bounded waits, on an mbarrier
 * that nothing arrives at (which = 0) or on a global flag that nothing sets
 * (which = 1).  The wait gives up after the library's limit (~2 s), the
 * kernel records its code in a fresh error word of its own and returns; the
 * call synchronises the device and writes that word to *code_out (0x102 for
 * the mbarrier, 0x104 for the flag).  The context stays usable; the
 * library's device error word is not touched.  Allocates 8 bytes of device
 * memory for the duration of the call.  Errors: CORA_EINVAL for a bad
 * argument or NULL code_out, CORA_ECUDA if a CUDA call fails. */
CORA_API int cora_check_wait_timeout(int32_t which, int32_t* code_out);

#ifdef __cplusplus
}
#endif

#endif /* CORA_H_ */
