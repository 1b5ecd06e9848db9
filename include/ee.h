/*
 * ee.h -- C ABI of libee: batch-1 decode of a frozen decoder-only transformer
 * with confidence-gated early exit, for NVIDIA GB300 (sm_103a).
 *
 * The method (arxiv 2609.14144, "One Size Does Not Fit All"):
 *   Section 2 / Section 4 step two: a readout -- a square d x d matrix plus an
 *     offset -- is applied to the residual stream after layer k; its result
 *     passes through the model's own final RMSNorm and unembedding unchanged.
 *   Section 2 / Section 4 step five: the confidence is the readout's top-1
 *     softmax probability; if it exceeds the deployment's threshold tau the
 *     readout's token is emitted, otherwise layers k+1..L and the LM head run
 *     and the full model's token is emitted.  An early token leaves the upper
 *     layers' key-value cache incomplete; the missing entries are supplied by
 *     projecting the exit-layer state through the upper layers' key and value
 *     matrices.
 *   Section 4 step three: more than one exit point is possible.
 *   Appendix B: decoding is greedy.
 *   Appendix C: the layer is four attention projections with grouped-query
 *     attention and a three-matrix gated feed-forward block.
 *
 * Conventions
 *   - Every function returns EE_OK (0) or a negative status; ee_last_error()
 *     returns a message for the calling thread's last failure.  No C++
 *     exception crosses this boundary.
 *   - Weights are bf16 bit patterns (uint16_t), row-major [out, in].
 *   - A context is not thread-safe; all its GPU work is enqueued on the
 *     stream given to ee_create, in order.
 *   - Numerics: weights bf16; activations (residual stream, normalised
 *     inputs, queries, scores, softmax, attention output, feed-forward
 *     product, readout output, logits) fp32; products of bf16 weights and fp32
 *     activations accumulate in fp32; the KV cache is bf16 (round to nearest
 *     even).  The gate compares fp32 p > fp32 tau (strict).  Argmax ties go
 *     to the lowest token id.  Where a tensor core multiplies an fp32 value
 *     (the decode step's attention scores; every product of the batched
 *     prompt and re-pass, EE_OPT_ROWS), the value enters as three bf16 parts
 *     whose sum is the value (24 significant bits), each part's products with
 *     bf16 operands exact in the fp32 accumulator.  Values handed between
 *     CTAs inside the persistent layer kernel keep all 32 bits.  Results
 *     therefore differ from a plain fp32 loop only in summation order.
 */
#ifndef EE_H_
#define EE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---------------------------------------------------- */
#define EE_OK 0
#define EE_EINVAL (-1)   /* bad argument (NULL, out-of-range id or size)      */
#define EE_ENOMEM (-2)   /* workspace too small / allocation failed           */
#define EE_ECUDA (-3)    /* a CUDA runtime call failed                        */
#define EE_ERANGE (-4)   /* the step(s) would pass max_ctx                    */
#define EE_EDEVICE (-5)  /* the device error word was set (NaN confidence,   */
                         /* token out of range, position overflow); sticky   */
                         /* until ee_reset                                    */
#define EE_ESTATE (-6)   /* call out of order (decode before prefill, weights */
                         /* missing, readout added after the first step)      */

#define EE_MAX_READOUTS 8

/* force argument of ee_decode_step / entries of a force schedule */
#define EE_FREE 0                       /* the gate decides               */
#define EE_FORCE_FULL 1                 /* never exit (gates still report) */
#define EE_FORCE_EXIT_AT(r) (2 + (r))   /* exit at readout r               */

/* where output arrays of ee_decode_n live */
#define EE_HOST 0
#define EE_DEVICE 1

typedef struct ee_ctx ee_ctx;

/* Model shape.  d_model, head_dim * n_heads and ffn_dim must be multiples of
 * 8; head_dim must be 64 or 128; n_heads a multiple of n_kv_heads with
 * n_heads / n_kv_heads <= 8.  max_ctx bounds every position; page_size is the
 * KV page length in positions (power of two, 16..256).  max_readouts <=
 * EE_MAX_READOUTS. */
typedef struct {
    int32_t n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn_dim, vocab;
    float rms_eps, rope_base;
    int32_t tied_embedding; /* 1: the LM head is the embedding matrix        */
    int32_t qkv_bias;       /* 1: Q, K and V projections carry biases        */
    int32_t max_ctx, page_size, max_readouts;
} ee_model_config;

/* Host-side bf16 weights, row-major [out, in].  Per-layer members are arrays
 * of n_layers pointers.  embed, final_norm and every layer tensor are
 * required; lm_head is ignored when tied_embedding is 1; bq/bk/bv only when
 * qkv_bias is 1.  Shapes: embed, lm_head [V, d]; norms [d]; wq [A*D, d];
 * wk, wv [K*D, d]; bq [A*D]; bk, bv [K*D]; wo [d, A*D]; wg, wu [F, d];
 * wd [d, F].  The caller keeps ownership; data are copied (and repacked)
 * into the workspace before ee_load_weights returns. */
typedef struct {
    const uint16_t* embed;
    const uint16_t* lm_head;
    const uint16_t* final_norm;
    const uint16_t* const* attn_norm;
    const uint16_t* const* wq;
    const uint16_t* const* wk;
    const uint16_t* const* wv;
    const uint16_t* const* bq;
    const uint16_t* const* bk;
    const uint16_t* const* bv;
    const uint16_t* const* wo;
    const uint16_t* const* mlp_norm;
    const uint16_t* const* wg;
    const uint16_t* const* wu;
    const uint16_t* const* wd;
} ee_host_weights;

/* Outcome of one gated step (Section 4, step five). */
typedef struct {
    int32_t token;        /* emitted token                                     */
    int32_t exited;       /* 1: emitted by a readout                           */
    int32_t exit_readout; /* index of that readout, or -1                      */
    int32_t exit_layer;   /* its layer, or n_layers for a full-depth step      */
    int32_t n_evaluated;  /* readouts evaluated this step                      */
    int32_t full_token;   /* LM head's token on full-depth steps, else -1      */
    int32_t gate_pass[EE_MAX_READOUTS];     /* p_r > tau_r at each evaluated r */
    int32_t readout_token[EE_MAX_READOUTS]; /* argmax of each evaluated readout */
    float confidence[EE_MAX_READOUTS];      /* p_r of each evaluated readout   */
    float full_confidence;                  /* LM head top-1 probability      */
    int32_t nucleus_member; /* EE_OPT_NUCLEUS on a full-depth step: 1 if readout 0's
                               token lies in the LM head's nucleus (Section 2
                               acceptance), else 0; -1 when not computed      */
    float nucleus_mass;     /* LM head probability of the tokens strictly more
                               probable than readout 0's token (0 if not computed) */
} ee_step_result;

/* Exit statistics since the last ee_reset (Section 2, "exit rate"). */
typedef struct {
    int64_t steps;                      /* gated decode steps                */
    int64_t full_steps;                 /* steps that ran all layers         */
    int64_t exits[EE_MAX_READOUTS];     /* steps emitted by each readout     */
} ee_stats;

/* ---- lifetime ---------------------------------------------------------- */

/* Device bytes a context with this shape needs: weights, readouts, paged KV
 * cache for max_ctx positions, activations and scratch. */
int ee_workspace_bytes(const ee_model_config* cfg, size_t* bytes);

/* Create a context on the current CUDA device.  d_workspace: device memory of
 * at least ee_workspace_bytes() bytes, 256-byte aligned, owned by the caller
 * and kept alive until ee_destroy; NULL makes the library allocate (and free)
 * it.  stream: a cudaStream_t (NULL = the legacy default stream) on which all
 * of the context's work is enqueued. */
int ee_create(const ee_model_config* cfg, void* d_workspace, size_t workspace_bytes, void* stream,
              ee_ctx** out);
int ee_destroy(ee_ctx* ctx);
const char* ee_last_error(void);

/* Upload and repack the frozen model (synchronous). */
int ee_load_weights(ee_ctx* ctx, const ee_host_weights* w);

/* Attach a readout after layer `layer` (1..n_layers): w [d, d] and b [d], bf16
 * (Section 2: a square matrix plus an offset).  Readouts must be added in
 * increasing layer order, before the first prefill.  *readout_id receives its
 * index (0-based), which selects its tau in every taus[] array. */
int ee_add_readout(ee_ctx* ctx, int layer, const uint16_t* w, const uint16_t* b, int* readout_id);

/* Map logical KV pages to physical pages: pages[i] in [0, n_pages) for the
 * ceil(max_ctx / page_size) logical pages, a permutation.  Default: identity.
 * Only between ee_reset and the next prefill. */
int ee_set_page_table(ee_ctx* ctx, const int32_t* pages, int n_pages);

/* Clear the KV cache marks, position, statistics and device error word. */
int ee_reset(ee_ctx* ctx);

/* ---- the hot path ------------------------------------------------------ */

/* Prefill n prompt tokens at full depth (no gate) from position 0, filling
 * the KV cache exactly; *first_token (may be NULL) receives the full model's
 * greedy token after the last prompt position, which is also kept on the
 * device as the next step's input.  Requires a fresh or reset context. */
int ee_prefill(ee_ctx* ctx, const int32_t* ids, int n, int32_t* first_token);

/* One gated decode step at the current position (Section 4, step five).
 * input_token in [0, V), or -1 for the token the previous call emitted.
 * taus: one threshold per readout (host array).  force: EE_FREE,
 * EE_FORCE_FULL or EE_FORCE_EXIT_AT(r); in forced modes every readout up to
 * the taken one (all of them for EE_FORCE_FULL) is still evaluated and its
 * gate verdict reported.  Synchronous: *out is filled before return. */
int ee_decode_step(ee_ctx* ctx, int32_t input_token, const float* taus, int force, ee_step_result* out);

/* n gated steps with the emitted token fed back on the device (one graph
 * launch, no host round trip between steps).  input_token as above.
 * force_schedule: NULL (the gate decides) or n host int8 entries with the
 * force values above (imposed exits).  tokens [n] int32, exit_readout [n]
 * int32 (-1 = full depth), confidence [n] float (p of the emitting readout,
 * or of the last evaluated readout on full steps; 0 with no readout); any may
 * be NULL.  where = EE_HOST: host arrays, the call returns after the results
 * are copied back; EE_DEVICE: device arrays of n entries, the call returns
 * once the work is enqueued. */
int ee_decode_n(ee_ctx* ctx, int n, int32_t input_token, const float* taus, const int8_t* force_schedule,
                int32_t* tokens, int32_t* exit_readout, float* confidence, int where);

/* Fidelity calibration pass (Section 2 acceptance; Section 4, step four).
 * n teacher-forced full-depth steps from the current position: step i takes
 * ids[i] as its input token, every readout is evaluated (its gate never
 * taken) and the LM head checks whether readout 0's token lies in the full
 * model's nucleus of share p_nuc, the smallest set of most probable tokens
 * whose probability reaches p_nuc: it does when the tokens strictly more
 * probable than it hold less than p_nuc.  One graph launch, no host round
 * trip between steps.
 *   ids    [n] int32 in [0, V)
 *   p_nuc  in (0, 1]
 *   conf   [n][n_readouts] float: each readout's confidence signal (the
 *          EE_OPT_CONFIDENCE kind) at step i, row-major; may be NULL
 *   member [n] int32: 1/0 nucleus membership of readout 0's token; may be NULL
 *   mass   [n] float: probability of the tokens above it; may be NULL
 *   where  EE_HOST: host arrays (ids read, results written before return);
 *          EE_DEVICE: device arrays, the call returns once enqueued.
 * The position advances by n; the KV cache holds the full model's entries of
 * ids and the next input is the full model's token after ids[n - 1].  The
 * steps count as full-depth steps in ee_get_stats.  Requires at least one
 * readout (EE_ESTATE otherwise); EE_EINVAL for a bad argument (ids are
 * range-checked on the host when where = EE_HOST, on the device otherwise:
 * an out-of-range id sets the device error word); EE_ERANGE if the steps
 * would pass max_ctx. */
int ee_calibrate(ee_ctx* ctx, const int32_t* ids, int n, float p_nuc, float* conf, int32_t* member, float* mass,
                 int where);

/* Full-depth re-pass over recent tokens (Section 11): every position t in
 * [t0, t1) whose upper-layer cache entries are still the fills of an early
 * exit runs those layers again, in position order, from the residual it
 * exited with (kept by the exit step), so that their entries become the ones
 * the full model computes given the cache before them (exactly the full
 * model's when every earlier exited position has been re-passed).  Positions
 * that ran at full depth are skipped.  The decode position and the next input
 * token are unchanged; the final hidden state read by EE_DBG_HIDDEN_FINAL is
 * the last re-passed position's.  *n_repassed (may be NULL) receives the number
 * of positions re-passed.  Synchronous.  EE_ERANGE unless 0 <= t0 <= t1 <=
 * position; EE_ESTATE before prefill.  See also EE_OPT_REPASS. */
int ee_repass(ee_ctx* ctx, int32_t t0, int32_t t1, int32_t* n_repassed);

/* Wait for the context's stream and report the device error word. */
/* Fill every key/value entry that EE_OPT_LAZY_FILL left pending: each
 * skipped layer's entry of each exited position becomes the projection of
 * the residual the position exited with (Section 4, step five), exactly as
 * the eager fill computes it.  Synchronous; EE_OK with nothing to do. */
int ee_flush_fills(ee_ctx* ctx);
int ee_sync(ee_ctx* ctx);
int ee_get_stats(ee_ctx* ctx, ee_stats* out);
/* Position of the next step's input token. */
int ee_position(ee_ctx* ctx, int32_t* pos);

/* ---- options and debug read-back -------------------------------------- */

#define EE_OPT_GRAPHS 1       /* 1 (default): CUDA graphs with conditional nodes;
                                 0: direct launches, branch decided on the host */
#define EE_OPT_PDL 2          /* 1 (default): programmatic dependent launch    */
#define EE_OPT_DEBUG_LOGITS 3 /* 1: keep each step's readout and final logits  */
#define EE_OPT_CONFIDENCE 5   /* the signal each gate compares with its tau: */
#define EE_CONF_PMAX 0        /*   top-1 probability p1 (Section 2; default)   */
#define EE_CONF_MARGIN 1      /*   p1 - p2, the margin to the second-best token */
#define EE_CONF_NEGENT 2      /*   sum_v p_v log p_v, the negative entropy (<= 0)
                                 (Section 10: the three are interchangeable);
                                 the step result's confidence reports it    */
#define EE_OPT_PERSISTENT 4   /* 1 (default where supported): each run of layers
                                 between readouts is one persistent launch, one
                                 CTA per SM streaming weights through a shared-
                                 memory ring; 0: five launches per layer.
                                 EE_EINVAL if the shape is not supported      */
#define EE_OPT_REPASS 7       /* 0 (default): off; P > 0: ee_decode_n re-passes
                                 (ee_repass) the P positions decoded since the
                                 last re-pass every P steps (Section 11's
                                 periodic full-depth pass); the call then
                                 synchronises at each re-pass              */
#define EE_OPT_NUCLEUS 6      /* 0 (default): off; 1..1000: full-depth steps of
                                 ee_decode_step report the nucleus membership of
                                 readout 0's token at share value/1000
                                 (Section 2 acceptance)                      */
#define EE_OPT_ROWS 8         /* 1: ee_prefill and ee_repass run each layer
                                 over batches of up to 256 positions, each
                                 weight read once per batch, each activation
                                 carried as three bf16 parts (24 significant
                                 bits), the projections on the tcgen05 tensor
                                 cores with TMA-staged operands (EE_EINVAL
                                 where unavailable); 2: the same batches with
                                 warp-level mma products; 0: one position
                                 at a time through the decode step's layer
                                 kernels (fp32 activations).  Default: 1
                                 where the tcgen05 path is available, else 0 */
#define EE_OPT_WAIT_LIMIT 9    /* for testing the failure path: the bound, in SM
                                 clock cycles, on each wait of the persistent
                                 layer kernel (ring stages, values from other
                                 CTAs); 0 (default): about 2 s.  A wait that
                                 runs out sets the device error word, the
                                 launch ends without waiting further (copies
                                 in flight still land first) and the call
                                 returns EE_EDEVICE; ee_reset clears it.  A
                                 few thousand cycles make ordinary waits run
                                 out.                                        */
#define EE_OPT_LAZY_FILL 11    /* 0 (default): an exit step fills the key/value
                                 entries of the layers it skips (Section 4,
                                 step five); 1: it only records the residual
                                 it exited with, and the next step that runs
                                 one of those layers first fills every such
                                 pending entry of the layers it runs (one read
                                 of their key/value weights for all pending
                                 positions).  Tokens are the same either way;
                                 ee_flush_fills fills what is still pending.
                                 Turning it off flushes.                     */
int ee_set_option(ee_ctx* ctx, int option, int value);

#define EE_DBG_HIDDEN_READOUT 1 /* layer = readout r: residual h_k it read, d floats   */
#define EE_DBG_READOUT_Y 2      /* layer = readout r: W_r h_k + b_r, d floats          */
#define EE_DBG_HIDDEN_FINAL 3   /* residual after layer L of the last full step        */
#define EE_DBG_READOUT_LOGITS 4 /* layer = readout r: V floats (EE_OPT_DEBUG_LOGITS)   */
#define EE_DBG_FINAL_LOGITS 5   /* V floats (EE_OPT_DEBUG_LOGITS)                      */
#define EE_DBG_KV 6             /* layer (0-based), pos: K then V, 2*K*D bf16          */
#define EE_DBG_KV_SRC 7         /* layer, pos: int8, 0 empty / 1 computed / 2 filled   */
/* Copy a piece of device state into host_dst (bytes must match exactly).
 * Synchronous. */
int ee_debug_read(ee_ctx* ctx, int what, int layer, int pos, void* host_dst, size_t bytes);

/* ---- measurement ------------------------------------------------------- */

#define EE_KERNEL_QKV 0      /* RMSNorm + Q/K/V GEMV + RoPE + KV append (one layer) */
#define EE_KERNEL_ATTN 1     /* split-K paged attention (one layer)                 */
#define EE_KERNEL_OPROJ 2    /* output projection + residual (one layer)            */
#define EE_KERNEL_GATEUP 3   /* RMSNorm + gate/up GEMV + SiLU product (one layer)   */
#define EE_KERNEL_DOWN 4     /* down projection + residual (one layer)              */
#define EE_KERNEL_READOUT 5  /* readout affine map                                  */
#define EE_KERNEL_VOCAB 6    /* unembedding pass with the confidence statistics     */
#define EE_KERNEL_KVFILL 7   /* KV fill of the layers above the first readout       */
#define EE_KERNEL_LAYERS 8   /* persistent kernel over layers 1..k (first readout);
                                0 when the shape does not support it               */
#define EE_NUM_KERNELS 9
/* Average device time (ms) of each decode kernel, from CUDA events around
 * `iters` back-to-back direct launches on the context's stream, cycling
 * through the layers so consecutive launches read different weights.  No
 * counterpart in the paper (measurement only).  Needs a prefilled context
 * with at least one readout; leaves the KV entries of the next position and
 * the residual scratch overwritten, which the next step rewrites anyway.
 * ms_out: host float[EE_NUM_KERNELS]. */
int ee_profile_kernels(ee_ctx* ctx, int iters, float* ms_out);

/* ---- standalone kernels on caller buffers ----------------------------- */

/* Split-K decode attention of one query position over a paged bf16 KV cache
 * (Section 2, "key-value cache"; grouped-query heads h -> h / (A / K)).
 *   q        device fp32 [A, D], already rotated
 *   k_pages, v_pages  device bf16 [n_pages, K, page_size, D]
 *   page_table device int32 [ceil(T / page_size)] logical -> physical page
 *   T        attended positions (1..)
 *   scratch  device fp32 workspace of ee_attention_scratch_bytes() bytes
 *   out      device fp32 [A, D] = softmax(q K^T / sqrt(D)) V
 * Enqueued on stream; returns without synchronising. */
int ee_attention_scratch_bytes(int n_heads, int n_kv_heads, int head_dim, size_t* bytes);
int ee_attention_decode(const float* q, const uint16_t* k_pages, const uint16_t* v_pages,
                        const int32_t* page_table, int T, int n_heads, int n_kv_heads, int head_dim,
                        int page_size, void* scratch, size_t scratch_bytes, float* out, void* stream);

/* Split-K decode attention for callers that cannot allocate device memory:
 * the same computation, arguments and result as ee_attention_decode, minus
 * the scratch buffer.  The paper has no counterpart; this exists for callers
 * whose device memory belongs entirely to another allocator, whose hot path
 * must not call cudaMalloc/cudaFree (which may synchronise the device), or
 * that have no allocator at all.
 *   Scratch lives in one fixed device area of EE_STATIC_ATTN_SCRATCH_BYTES
 *   inside this library, held by every GPU that loads the library until the
 *   process exits.  Shapes needing more (n_heads * (head_dim + 2) above about
 *   4096) are rejected with EE_EINVAL and a message.
 *   The area is shared by every call and keeps the previous call's contents;
 *   each call clears the part that must start at zero.  Calls whose work
 *   overlaps on the GPU (other streams, other threads) race on the area:
 *   order them on one stream.
 *   Every call looks up the area's device address on the current device
 *   (so an address never outlives a cudaDeviceReset); the first call on a
 *   device also loads the library's device code there, so make that first
 *   call before any stream capture.
 *   No cudaMalloc, cudaFree or other allocating call is made. */
#define EE_STATIC_ATTN_SCRATCH_BYTES (2u << 20)
int ee_attention_decode_static(const float* q, const uint16_t* k_pages, const uint16_t* v_pages,
                               const int32_t* page_table, int T, int n_heads, int n_kv_heads, int head_dim,
                               int page_size, float* out, void* stream);

/* One pass over an unembedding matrix with the readout's confidence test
 * (Section 2 readout + confidence gate; Section 4 step five):
 *   x        device fp32 [d] residual-space vector (a readout output or h_L)
 *   gain     device bf16 [d] final RMSNorm gain;  U device bf16 [V, d]
 *   z = RMSNorm(x) * gain;  l = U z;  p = 1 / sum_v exp(l_v - max l)
 *   out_token device int32[1] (lowest argmax), out_p device float[1]
 *   logits   device fp32 [V] or NULL
 *   scratch  device workspace of ee_vocab_scratch_bytes() bytes
 * Enqueued on stream. */
int ee_vocab_scratch_bytes(int vocab, int d_model, size_t* bytes);
int ee_vocab_confidence(const float* x, const uint16_t* gain, const uint16_t* U, int vocab, int d_model,
                        float eps, void* scratch, size_t scratch_bytes, int32_t* out_token, float* out_p,
                        float* logits, void* stream);
/* The same pass returning all three confidence signals of Section 10:
 *   out_signals device float[3] = { p1, p1 - p2, sum_v p_v log p_v }
 * where p2 is the second-best probability (p1 again if the maximum is tied).
 * Other arguments and errors as for ee_vocab_confidence. */
int ee_vocab_signals(const float* x, const uint16_t* gain, const uint16_t* U, int vocab, int d_model,
                     float eps, void* scratch, size_t scratch_bytes, int32_t* out_token, float* out_signals,
                     float* logits, void* stream);

/* Threshold selection (Section 4, step four): the lowest tau at which at
 * least a share `target` of the early answers (the positions with
 * conf > tau) are acceptable.  Candidates are -inf (every position exits)
 * and each conf[i * conf_stride]; a candidate with no early answer does not
 * count; *tau = +inf when no candidate reaches the target.  The acceptance
 * test is good >= target * early in double precision.
 *   conf    device float, n entries at stride conf_stride (>= 1), e.g. one
 *           column of ee_calibrate's conf
 *   member  device int32 [n], nonzero = acceptable
 *   target  in [0, 1]
 *   tau     device float [1] (result)
 *   scratch device workspace of 8 bytes
 * Enqueued on stream (n >= 1; EE_EINVAL otherwise).  The work is n + 1
 * candidates times n comparisons, spread over the whole GPU. */
int ee_select_tau(const float* conf, int conf_stride, const int32_t* member, int n, float target, float* tau,
                  void* scratch, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* EE_H_ */
