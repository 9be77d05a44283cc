/*
 * ssd.h - C ABI of libssd: batch-1 self-speculative decoding on one GB300.
 *
 * Method: Zhang et al., "Draft & Verify: Lossless Large Language Model
 * Acceleration via Self-Speculative Decoding" (arxiv 2309.08168).
 *   - Drafting (Sec. 3.2, Algorithm 2): the model drafts K tokens with a set
 *     of attention / MLP sublayers skipped (the vector z of Sec. 3.3, Eq. 1).
 *   - Verification (Algorithm 2 / Algorithm 4): one forward of the full model
 *     over the K+1 positions [x_last, d_1..d_K]; greedy: the longest prefix of
 *     drafts equal to the target's argmax is accepted and the first mismatch
 *     corrected (or a bonus token added); sampling: draft d_j is accepted
 *     when r < min(1, p/q), the first rejected one is resampled from
 *     norm(max(0, p - q)), a bonus is sampled from p when all are accepted.
 *   - KV rollback: the committed cache length becomes len + 1 + n, where n is
 *     the number of accepted drafts.
 *
 * Conventions for every call:
 *   - Return value: SSD_OK (0) or a negative SSD_ERR_* code; the message of
 *     the last failure on the calling thread is in ssd_last_error().
 *   - A handle is bound to one CUDA device (the current one at ssd_create)
 *     and one stream; calls on one handle must not run concurrently.
 *   - Host outputs are complete when the call returns.
 *   - All matrices are bf16, row-major [out_features][in_features] (the
 *     Hugging Face LLaMA layout); norm gains are bf16 vectors.
 */
#ifndef SSD_H
#define SSD_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SSD_OK 0
#define SSD_ERR_INVALID_ARG (-1) /* bad pointer, size or configuration */
#define SSD_ERR_OOM (-2)         /* device memory allocation failed */
#define SSD_ERR_CUDA (-3)        /* a CUDA call or kernel failed */
#define SSD_ERR_CAPACITY (-4)    /* prompt + n_new exceeds max_seq */
#define SSD_ERR_TIMEOUT (-5)     /* a bounded device wait gave up (a grid barrier or a copy that did not
                                    complete within its limit); the handle stays usable */
#define SSD_ERR_STATE (-6)       /* call out of order (e.g. generate without a prompt or prefill) */

typedef struct ssd_handle ssd_handle;

/* Model shape (LLaMA-2 decoder, Sec. 4.1 / App. B).
 *   head_dim must be 64 or 128; n_heads a multiple of n_kv_heads (GQA);
 *   d_model, n_heads * head_dim and n_kv_heads * head_dim multiples of 128
 *   (the forward kernel's 128-row tiles); ffn a multiple of 16 and >= 64;
 *   2 <= vocab <= 32768;
 *   max_seq = KV capacity in positions (>= n_prompt + n_new).
 * Numerics: bf16 weights; fp32 residual stream, norms, softmax and
 * accumulation; activations enter each projection as bf16 hi + lo pairs;
 * fp16 KV cache; fp32 logits. */
typedef struct {
    int n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn, vocab, max_seq;
    float rms_eps, rope_theta;
} ssd_config;

/* Model weights.  Per-layer members point to HOST arrays of n_layers
 * pointers.  on_device = 1: the tensor pointers are device pointers on the
 * handle's device; they are borrowed (not copied) and must stay valid and
 * unchanged until ssd_destroy.  on_device = 0: they are host pointers; the
 * library copies them into device memory it owns, and the caller may free
 * them when ssd_create returns.
 * Shapes: embed, lm_head [vocab][d]; wq [H*hd][d]; wk, wv [Hkv*hd][d];
 * wo [d][H*hd]; w_gate, w_up [ffn][d]; w_down [d][ffn]; norms [d]. */
typedef struct {
    const void* embed;
    const void* final_norm;
    const void* lm_head;
    const void* const* wq;
    const void* const* wk;
    const void* const* wv;
    const void* const* wo;
    const void* const* attn_norm;
    const void* const* w_gate;
    const void* const* w_up;
    const void* const* w_down;
    const void* const* mlp_norm;
    int on_device;
} ssd_weights;

typedef enum { SSD_GREEDY = 0, SSD_SAMPLE = 1 } ssd_mode;

/* Acceptance statistics of one ssd_generate call (the paper's acceptance
 * rate AR of Sec. 3.4 is accepted / drafted). */
typedef struct {
    int rounds;        /* draft + verify rounds */
    int drafted;       /* draft tokens produced */
    int accepted;      /* draft tokens accepted */
    int emitted;       /* tokens written to out_tokens (== n_new) */
    double accept_rate;/* accepted / drafted (0 when nothing was drafted) */
    int hist[33];      /* hist[n] = rounds that accepted n drafts */
    float draft_ms;    /* GPU time in drafting stages (CUDA events) */
    float verify_ms;   /* GPU time in verification stages incl. acceptance */
    float total_ms;    /* GPU time of the decode loop (prefill excluded) */
    long long kernel_launches; /* CUDA kernels launched by the decode loop */
    float gamma;       /* draft-exit threshold after the last round (0 when the exit is off) */
} ssd_stats;

/* Creates a handle: validates the shape, takes the weights (see
 * ssd_weights), allocates the KV cache (2 * n_layers * n_kv_heads * max_seq *
 * head_dim fp16) and work buffers on the current device.  cuda_stream: a
 * cudaStream_t to run on, or NULL for a stream the handle creates.  The skip
 * set starts empty (draft = full model); sampling starts at temperature 1,
 * top_p 1.  Errors: INVALID_ARG, OOM, CUDA. */
int ssd_create(const ssd_config* cfg, const ssd_weights* weights, void* cuda_stream,
               ssd_handle** out);

/* Sets the draft model's skip set z (Sec. 3.3, Eq. 1): mask[2l] = 1 skips
 * the attention sublayer of layer l, mask[2l+1] = 1 its MLP sublayer; a
 * skipped sublayer adds nothing to the residual stream and (attention) reads
 * and writes no KV.  n_sublayers must equal 2 * n_layers; values must be 0 or
 * 1.  The mask is copied.  Errors: INVALID_ARG. */
int ssd_set_skip(ssd_handle* h, const uint8_t* mask, int n_sublayers);

/* Sampling parameters for SSD_SAMPLE (App. B, Table "Hyperparameter
 * settings"): p = softmax(logits / temperature) restricted to the nucleus
 * {x : p(x) >= tau*} holding at least top_p of the mass, renormalised; the
 * same transform gives the draft distribution q.  temperature > 0,
 * 0 < top_p <= 1.  Errors: INVALID_ARG. */
int ssd_set_sampling(ssd_handle* h, float temperature, float top_p);

/* Adaptive draft exit (Sec. 3.4, Eqs. 2-4; Algorithms 3 / 4 of App. G).
 * enable = 1: within a round, the draft whose confidence - the largest
 * probability of the distribution it was chosen from (softmax of the draft
 * logits in greedy mode, the temperature / nucleus distribution in sampling
 * mode) - falls below gamma is the round's last draft (it is still
 * verified).  After every verification that had drafts, with AR_e =
 * accepted / drafted of that round:
 *   AR <- beta1 AR + (1 - beta1) AR_e       (beta1 = 0 at the first update)
 *   gamma <- beta2 gamma + (1 - beta2) (gamma + eps if AR <= alpha, else gamma - eps)
 * gamma starts at gamma0 in every ssd_generate call; beta2 = 1 keeps a static
 * threshold.  enable = 0 (the default) drafts K tokens every round (Alg. 2).
 * The exit keeps greedy output identical to autoregressive output.  Needs
 * gamma0 >= 0, eps >= 0 and alpha, beta1, beta2 in [0, 1].
 * Errors: INVALID_ARG. */
int ssd_set_draft_exit(ssd_handle* h, int enable, float gamma0, float alpha, float eps, float beta1,
                       float beta2);

/* Prefill: encodes the prompt with the full model before decoding starts
 * (Sec. 3.1: the prefix x_1..x_t that Algorithms 1 and 2 continue from).
 * It runs prompt[0 .. n_prompt-2] through the full model, filling KV
 * positions [0, n_prompt-1); prompt[n_prompt-1] becomes the first round's
 * x_last, so every generated token comes from a decoding round.  prompt is a
 * host array of token ids in [0, vocab); 1 <= n_prompt <= max_seq.
 * Errors: INVALID_ARG, CAPACITY, CUDA, TIMEOUT. */
int ssd_prefill(ssd_handle* h, const int32_t* prompt, int n_prompt);

/* Generates n_new tokens (Algorithm 2 for SSD_GREEDY, Algorithm 4 for
 * SSD_SAMPLE) with K drafts per round; K = 0 is plain autoregressive
 * decoding (Algorithm 1) through the same verification kernels.  The last
 * round drafts min(K, remaining - 1) tokens.  If prompt != NULL it is
 * prefilled first; if prompt == NULL decoding restarts from the state right
 * after the last ssd_prefill (the prompt's KV is kept).  seed keys the
 * Philox4x32-10 stream of SSD_SAMPLE.  out_tokens: host array of n_new ids.
 * stats may be NULL.  0 <= K <= 15; n_prompt + n_new <= max_seq.
 * Errors: INVALID_ARG, CAPACITY, STATE, CUDA. */
int ssd_generate(ssd_handle* h, const int32_t* prompt, int n_prompt, int n_new, int K,
                 ssd_mode mode, uint64_t seed, int32_t* out_tokens, ssd_stats* stats);

/* Parity hook: one forward of n_rows tokens (host ids) at positions
 * pos0 .. pos0+n_rows-1 over the current KV cache, full model (draft = 0:
 * the verification forward of Algorithm 2 / 4, which produces the target
 * rows p_0..p_K) or the skip-set model (draft = 1: one drafting step of
 * Sec. 3.2, the draft distribution q), writing KV like the decode loop does
 * and copying fp32 logits [n_rows][vocab] to host logits_out.
 * 1 <= n_rows <= 16; pos0 + n_rows <= max_seq.
 * Errors: INVALID_ARG, CUDA, TIMEOUT. */
int ssd_debug_forward(ssd_handle* h, int draft, const int32_t* tokens, int n_rows, int pos0,
                      float* logits_out);

/* Test hook for the bounded waits (the paper has no counterpart): arms the
 * next ssd_debug_forward on this handle to make its grid barrier number
 * `barrier` (1 = the barrier after the embedding) unreachable and to give up
 * waiting after wait_limit_s seconds; that forward then returns
 * SSD_ERR_TIMEOUT, its logits are unspecified and the handle stays usable
 * (the next forward runs normally).  barrier = 0 disarms.  The hook applies
 * to that one forward only, never to ssd_generate or ssd_prefill.
 * 0 < wait_limit_s <= 10.  Errors: INVALID_ARG. */
int ssd_debug_stall_barrier(ssd_handle* h, int barrier, double wait_limit_s);

/* Parity hook for the speculative-sampling acceptance kernel of Algorithm 4
 * in isolation: `trials` independent verifications sharing the target rows
 * p (host fp32, (Kd+1) x vocab, each row a distribution) and draft rows q
 * (host fp32, Kd x vocab); trial t uses drafts[t*Kd .. t*Kd+Kd-1] (host) and
 * the Philox stream of seeds[t] at positions pos0 + 1 ...; it writes
 * out[2t] = accepted count n and out[2t+1] = the correction / bonus token.
 * 1 <= Kd <= 15.  Errors: INVALID_ARG, OOM, CUDA. */
int ssd_debug_spec_accept(ssd_handle* h, const float* p, const float* q, int Kd,
                          const int32_t* drafts, const uint64_t* seeds, int trials, int pos0,
                          int32_t* out);

/* Profiling hook: captures one forward over `rows` rows at the last `rows`
 * positions of the KV cache (full model, or the skip-set model if draft)
 * into a CUDA graph, replays it `reps` times on the handle's stream between
 * two CUDA events, and writes the average time of one forward (ms), the
 * number of kernels in it and the weight bytes it streams from HBM.  With
 * gemm_only = 1 the time, count and bytes cover the projection ops only
 * (their share of one replay, read from the forward kernel's device trace).
 * KV positions [max_seq - rows, max_seq) are overwritten: if they reach into
 * the prefilled prompt, the next ssd_generate needs a prompt again.
 * 1 <= rows <= 16, reps >= 1.  Errors: INVALID_ARG, CUDA. */
int ssd_debug_time_forward(ssd_handle* h, int draft, int rows, int gemm_only, int reps,
                           float* ms_per_forward, int* launches, double* weight_bytes);

/* Profiling hook: one forward as in ssd_debug_time_forward, with the device
 * trace of the forward kernel: op_us[o] = microseconds of op o (from the end
 * of op o-1 to the end of op o, grid barrier included), op_types[o] = 0
 * embedding, 1 q/k/v projection, 2 attention, 3 output or down projection,
 * 4 gate/up projection, 5 lm_head.  max_ops >= 2 + 5 * n_layers is always
 * enough.  detail_op: -1 (none), or the index of one op to trace in detail
 * plus 65536 x the CTA whose unit stamps are taken (0 for CTA 0).
 * unit_trace (may be NULL): 256 globaltimer stamps (ns) of that CTA for
 * that op.  A projection: its first 64 work units, 4 per unit: producer
 * issue, MMAs issued, 0, segment flush done (0 if none).
 * Attention: its first 31 items, 8 per item: item start, q loaded, K / V
 * ready, after the CTA barrier, scores done, softmax done, P V done, 0.
 * cta_trace (may be NULL): 8 stamps per CTA of the forward kernel for
 * detail_op: [0] op start, [1] first data ready (attention), [2] last
 * accumulator ready (projections) or arrival at the grid barrier between the
 * segment partials and their combine (attention), [3] work done, [4] grid
 * barrier arrive, [5] barrier release, [6] number of work units (items),
 * [7] release of the attention's inner grid barrier (0 for projections);
 * max_ctas >= the grid (the SM count), *n_ctas = the grid.
 * Errors: INVALID_ARG, CUDA. */
int ssd_debug_trace_forward(ssd_handle* h, int draft, int rows, float* op_us, int* op_types,
                            int max_ops, int* n_ops, int detail_op, unsigned long long* unit_trace,
                            unsigned long long* cta_trace, int max_ctas, int* n_ctas);

/* Allocation-free projection.  The paper has no counterpart: this is a
 * service of this library for callers that cannot allocate device memory
 * when they need a projection, e.g. a serving process that reserves all of
 * HBM at start-up and treats any later allocation as an error, a plug-in
 * whose host framework owns every device allocation, or a latency-critical
 * loop that must not call cudaMalloc / cudaFree because they can synchronise
 * the device.  It runs the decoder's projection GEMM kernel alone:
 *     y[m][n] = sum_k x[m][k] * w[n][k],   m < M, n < N,
 * w: device bf16 [N][K] row-major; x: device fp32 [M][K] (entering the MMA
 * as bf16 hi + lo pairs, as inside the decoder); y: device fp32 [M][N]; all
 * owned by the caller; w and x 16-byte aligned.  1 <= M <= 16, K a positive
 * multiple of 16.  cuda_stream: the stream to launch on (NULL = legacy
 * default stream); the call returns after enqueueing the work.
 * Scratch: nothing is allocated.  The split-K partial sums and the per-tile
 * arrival counters live in fixed device arrays of the library, 1,048,576
 * floats and 4,096 counters (about 4 MiB per GPU that loads the library,
 * held until the process exits).  A problem needs ceil(N/64) <= 4096 tiles
 * and, when K > 512, ceil(K/512) * M * 64 * ceil(N/64) <= 1,048,576 scratch
 * floats; larger problems are rejected with SSD_ERR_CAPACITY before any
 * launch.  The first call on each device does a one-time set-up with that
 * device current (symbol lookup, kernel attribute); make that first call
 * before any stream capture.  Every call zeroes the counters it uses on the
 * stream before its kernel; the scratch arrays are shared by all calls on a
 * device, so calls that overlap on the GPU (other streams, other threads)
 * race and must be serialised by the caller.  Faults inside the kernel are
 * not reported by this call (it returns once the work is enqueued); builds
 * with the device-side checks enabled (SSD_CHECKED=1) read the check flag
 * back after the kernel, which makes the call synchronous, and report a
 * failed check as SSD_ERR_CUDA.
 * Errors: INVALID_ARG, CAPACITY, CUDA. */
int ssd_linear_noalloc(const void* w, const float* x, float* y, int N, int K, int M,
                       void* cuda_stream);

/* Releases everything the handle owns (never the borrowed weights). */
void ssd_destroy(ssd_handle* h);

/* Message of the last failure on this thread ("" if none). */
const char* ssd_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* SSD_H */
