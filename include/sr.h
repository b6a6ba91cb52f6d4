/*
 * libsr -- Speculative Rejection (Sun et al., "Fast Best-of-N Decoding via
 * Speculative Rejection", arXiv 2410.20290) on one GB300 GPU (sm_103a).
 *
 * The library generates N candidate responses to one prompt with a generator
 * transformer p, runs rejection rounds in which a reward model s scores every
 * partial response, cuts the batch at the alpha-quantile of those partial
 * rewards and compacts the survivors, and returns the highest-reward
 * completed response (Algorithm 1, Section 4.2).  alpha = 0 is Best-of-N
 * (Section 5.1).
 *
 * Conventions for every entry point:
 *   - No exception crosses this boundary.  Each call returns an sr_status; on
 *     failure sr_last_error() returns a thread-local message describing it.
 *   - The caller owns every buffer it passes.  Host pointers may be freed as
 *     soon as the call returns.  The library copies weights into its own
 *     device memory at sr_init and owns them, the KV page pool and all
 *     workspace until sr_destroy.
 *   - After SR_ERR_CUDA or SR_ERR_TIMEOUT the context must be destroyed.
 *   - Results are a pure function of (weights, prompt, arguments, seed):
 *     random draws are keyed on (seed, candidate id, token index).
 *   - "stream" arguments are cudaStream_t values passed as void*; NULL means
 *     the context's own stream (sr_k_* calls: the legacy default stream).
 */
#ifndef SR_H
#define SR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SR_OK = 0,
  SR_ERR_INVALID_ARG = 1, /* argument outside the documented range; nothing was run */
  SR_ERR_OOM = 2,         /* device allocation failed, or the KV pool cannot hold the next step */
  SR_ERR_CUDA = 3,        /* a CUDA call failed; the context is unusable */
  SR_ERR_TIMEOUT = 4,     /* a device-side wait hit its iteration limit; the context is unusable */
  SR_ERR_STATE = 5,       /* call out of order (e.g. a step on a finished batch) */
  SR_ERR_UNSUPPORTED = 6  /* a shape the kernels are not built for (see sr_init) */
} sr_status;

enum { SR_NORM_RMS = 0, SR_NORM_LAYER = 1 };
enum { SR_ACT_SWIGLU = 0, SR_ACT_GELU = 1, SR_ACT_GEGLU = 2 };
enum { SR_POS_ROPE = 0, SR_POS_LEARNED = 1 };
enum { SR_DT_F32 = 0, SR_DT_BF16 = 1, SR_DT_F16 = 2 };
enum { SR_SCHED_FIXED = 0, SR_SCHED_POOL_FULL = 1 };

/*
 * Shape of a decoder-only transformer (the generator p or the reward model s
 * of Section 3).  Weight blob layout (all tensors of type `dtype`, densely
 * packed in this order, matrices [out_features][in_features] row-major):
 *   tok_emb [vocab][d]; pos_emb [max_pos][d] (pos == LEARNED only);
 *   per layer: attn_norm_w [d]; attn_norm_b [d] (LAYER only);
 *              wqkv [(n_heads + 2 n_kv_heads) head_dim][d] (q rows, then k, then v);
 *              wo [d][n_heads head_dim]; mlp_norm_w [d]; mlp_norm_b [d] (LAYER only);
 *              gated act: w_gate [ffn][d], w_up [ffn][d]; GELU: w_fc [ffn][d];
 *              w_down [d][ffn];
 *   final_norm_w [d]; final_norm_b [d] (LAYER only);
 *   lm_head [vocab][d] (has_lm_head); score_head [d] (has_scalar_head).
 * Linear layers have no bias.  RoPE uses rotate-half pairing.  window > 0
 * limits attention to the last `window` positions.
 */
typedef struct {
  int n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn_dim, vocab, max_pos, window;
  int norm; /* SR_NORM_* */
  int act;  /* SR_ACT_* */
  int pos;  /* SR_POS_* */
  float rope_theta, norm_eps;
  int has_lm_head, has_scalar_head;
  int dtype; /* SR_DT_*: type of the weight blob.  SR_DT_F32 models compute in fp32 on the CUDA cores;
                SR_DT_BF16 / SR_DT_F16 models run fp16 operands and KV cache on the tensor cores with
                fp32 accumulation (bf16 weights of magnitude >= 2^-17 are exact in fp16). */
} sr_model_desc;

/*
 * Decision schedule (Algorithm 1, the generate-until-tau line, and Section
 * 4.2 "Early Generation").  FIXED: a rejection round runs when the live
 * candidates have generated tau[i] tokens, for each of the n_tau ascending
 * values.  POOL_FULL: a round runs before any decode step for which the KV
 * page pool cannot give every live candidate the page it needs (the
 * memory-triggered rounds of Section 4.2); tau is ignored.
 */
typedef struct {
  int kind; /* SR_SCHED_* */
  int n_tau;
  const int* tau; /* host array, n_tau ascending values >= 1 */
} sr_schedule;

/* Kernel classes timed when profiling is on (sr_set_profiling). */
enum {
  SR_KC_GEMM_DECODE = 0,  /* generator projections + LM head during decode (tcgen05 / fp32 GEMM) */
  SR_KC_GEMM_SCORE = 1,   /* reward-model projections while scoring partial / final responses */
  SR_KC_GEMM_PROMPT = 2,  /* prompt prefill projections (both models) */
  SR_KC_ATTN_DECODE = 3,  /* paged GQA decode attention (+ split combine) */
  SR_KC_ATTN_PREFILL = 4, /* prefill attention (prompt and scoring) */
  SR_KC_SAMPLE = 5,       /* Gumbel-max sampling */
  SR_KC_ELEMENTWISE = 6,  /* embedding, norms, RoPE + KV append, activations, score head, page copies */
  SR_KC_CONTROL = 7,      /* page allocation / release, rejection round, compaction, final argmax */
  SR_KC_N = 8
};

#define SR_MAX_ROUNDS 64
/* Per-call statistics of sr_generate (host struct filled by the library). */
typedef struct {
  int rounds;                             /* rejection rounds run */
  int b_per_round[SR_MAX_ROUNDS];         /* batch size b scored in round r (Eq. partial.reward.set) */
  int step_per_round[SR_MAX_ROUNDS];      /* tokens generated by live candidates when round r ran (tau) */
  int k_per_round[SR_MAX_ROUNDS];         /* order-statistic index used for r_cut */
  int accepted_per_round[SR_MAX_ROUNDS];  /* |I_accepted| of round r */
  float r_cut_per_round[SR_MAX_ROUNDS];   /* r_cut of round r (Eq. cutoff.threshold) */
  int k_raised;                           /* rounds whose k was raised to free enough pages */
  int n_completed;                        /* |I| */
  int best_id;                            /* candidate id k* of the returned response */
  int waves;                              /* pool-sized Best-of-N waves (alpha = 0 with POOL_FULL), else 1 */
  long long gen_tokens;                   /* tokens sampled from the generator */
  long long rm_tokens;                    /* positions run through the reward model: the prompt once, then every
                                             scored response position not read from the reward-model cache */
  long long decode_steps;                 /* batched decode steps */
  int pool_pages;                         /* pages in the KV pool */
  int peak_pages_in_use;
  double ms_prefill, ms_decode, ms_score, ms_select, ms_total; /* wall-clock phases, stream-synchronised */
  /* per kernel class (zero unless profiling is on): launch count and algorithmic work of all
     launches -- 2 M N K flops for a GEMM, 4 dh (keys) flops per query head for attention; bytes =
     operands read + results written once (decode attention: the shared prompt KV once plus each
     candidate's own KV) -- and, for the launches timed with CUDA events on the context's stream
     (all of them, or one in `period`, see sr_set_profiling), their count, summed time and work */
  double kern_ms[SR_KC_N];          /* summed event time of the timed launches */
  long long kern_launches[SR_KC_N]; /* all launches */
  double kern_flops[SR_KC_N];       /* all launches */
  double kern_bytes[SR_KC_N];       /* all launches */
  long long kern_timed[SR_KC_N];    /* timed launches */
  double kern_timed_flops[SR_KC_N];
  double kern_timed_bytes[SR_KC_N];
  long long rm_tokens_cached;  /* scored response positions whose reward-model K/V came from the cache
                                  (sr_set_rm_cache) instead of being run again */
} sr_stats;

typedef struct sr_ctx sr_ctx;
typedef struct sr_batch sr_batch;

/*
 * sr_init -- create a context on `device`.
 *   gen, gen_w : generator descriptor and weight blob (host or device pointer,
 *                copied with cudaMemcpyDefault under unified addressing; not retained).
 *                gen->has_lm_head must be 1.
 *   rm, rm_w   : reward-model descriptor and blob; rm->has_scalar_head must be 1.
 *                gen and rm must use the same vocabulary and dtype.
 *   kv_pool_bytes : generator KV-cache pool size in bytes (Section 5 "Setup":
 *                the KV cache is pre-allocated to what fits).  0 sizes the
 *                pool at each sr_generate to hold all N candidates to max_new.
 *   page_tokens : positions per page; must be 16.
 * Supported shapes: head_dim in {32, 64, 128, 256} (decode attention: 32, 64,
 * 128), n_heads % n_kv_heads == 0 with group size in {1, 2, 4, 8}, d_model %
 * 64 == 0, ffn_dim % 64 == 0, vocab % 32 == 0 for bf16 models.
 * Errors: SR_ERR_INVALID_ARG, SR_ERR_UNSUPPORTED, SR_ERR_OOM, SR_ERR_CUDA.
 */
sr_status sr_init(sr_ctx** out, const sr_model_desc* gen, const void* gen_w, const sr_model_desc* rm,
                  const void* rm_w, size_t kv_pool_bytes, int page_tokens, int device);
void sr_destroy(sr_ctx* ctx);
const char* sr_last_error(void);
/* Use `stream` (a cudaStream_t) for all later work of this context; NULL restores the context's stream. */
sr_status sr_set_stream(sr_ctx* ctx, void* stream);
/* b_init of Algorithm 1's first step ("based on the GPU memory capacity and the prompt length"): the
 * largest N <= n_max whose candidates can all generate tau_min tokens in a pool of kv_pool_bytes (pages
 * as in sr_init: floor(bytes / (16 positions x KV bytes per position of `gen`))) before the first
 * memory-triggered round -- pages - floor(P / 16) shared prompt pages, divided by the private pages one
 * candidate holds after tau_min tokens.  Host-only arithmetic.  *n_out gets the value (0 when nothing fits).
 * Errors: SR_ERR_INVALID_ARG (null or non-positive argument), SR_ERR_OOM (*n_out = 0). */
sr_status sr_auto_b_init(const sr_model_desc* gen, size_t kv_pool_bytes, int P, int tau_min, int n_max,
                         int* n_out);

/* Reward used by the rejection rounds and the final choice (Eq. partial.reward.set, Eq. output.SBoN):
 *   SR_REWARD_MODEL   the reward model s of sr_init (default);
 *   SR_REWARD_LOGPROB the self-likelihood objective of Section 5.3, s(Y) = ln p(Y | X) / len(Y)
 *                     under the generator itself (softmax of the raw logits: temperature 1, no EOS
 *                     bias), a partial response scored over its tau tokens.  The sampler keeps
 *                     ln p per candidate in the same pass over the logits; no reward-model work
 *                     runs (sr_stats.rm_tokens = 0).
 * The kind is read when a batch starts (sr_generate, sr_batch_begin); errors: SR_ERR_INVALID_ARG. */
enum { SR_REWARD_MODEL = 0, SR_REWARD_LOGPROB = 1 };
sr_status sr_set_reward(sr_ctx* ctx, int kind);
/* Reward-model KV kept across rejection rounds.  A partial reward s(X ++ Y^{<=tau}) (Eq.
 * partial.reward.set) needs the reward model's keys and values of every position before the last; the
 * paper re-runs them at every round and at the final score, the cost Section 1 calls quadratic.  With
 * `bytes` > 0 the library keeps, in a second paged pool of floor(bytes / (16 x the reward model's KV bytes
 * per position)) pages, each candidate's reward-model K/V of the response positions it has scored; a later
 * round, or the final score of a survivor, runs only the positions added since and attends to the cached
 * ones.  At a round, the batch's new positions go into the pool for every candidate (ascending id) whose
 * pages the free pool can still give; the others are scored in full as without the cache.  Rejected and
 * finished candidates' pages return to the pool when the next scoring starts.  Results agree with full
 * rescoring up to floating-point summation order.  0 (the default) turns it off.  Read when a batch starts
 * (sr_generate, sr_batch_begin); a context holds the pool until sr_destroy or a call with bytes = 0.
 * The prompt's reward-model KV is always computed once per batch.  Errors: SR_ERR_INVALID_ARG (null ctx);
 * SR_ERR_OOM at the next sr_generate / sr_batch_begin when the pool cannot be allocated. */
sr_status sr_set_rm_cache(sr_ctx* ctx, size_t bytes);
/* Per-kernel-class CUDA-event timing: 0 off; k >= 1 times one launch in k of each class (1: every
   launch; each timed launch adds two event records to the stream) and counts all of them.  Results
   land in sr_stats.kern_*.  Errors: SR_ERR_INVALID_ARG (null context, k < 0). */
sr_status sr_set_profiling(sr_ctx* ctx, int enable);

/*
 * sr_generate -- Algorithm 1 end to end for one prompt (host buffers).
 *   prompt [P] token ids (host), 1 <= P, P + max_new <= min(gen->max_pos, rm->max_pos).
 *   N      initial batch b_init (Algorithm 1, first line), 1 <= N <= 4096.
 *   alpha  rejection rate in [0, 1] (Eq. cutoff.threshold); 0 is Best-of-N.
 *   sched  decision schedule (see sr_schedule).
 *   max_new  cap on generated tokens; a candidate completes at EOS or max_new.
 *   temperature > 0; eos_bias is added to the EOS logit before temperature;
 *   eos_id in [0, vocab) or -1 for none.
 *   seed   key of the Philox4x32-10 noise.
 * Outputs (host): out_tokens [max_new] (the returned response Y_SR, Eq.
 * output.SBoN), *out_len its length, *out_score its reward s(Y_SR); st may be NULL.
 * Errors: SR_ERR_INVALID_ARG, SR_ERR_OOM (pool cannot hold the prompt tails or a
 * step even after raising k), SR_ERR_CUDA, SR_ERR_TIMEOUT.
 */
sr_status sr_generate(sr_ctx* ctx, const int32_t* prompt, int P, int N, float alpha, const sr_schedule* sched,
                      int max_new, float temperature, float eos_bias, int eos_id, uint64_t seed, int32_t* out_tokens,
                      int* out_len, float* out_score, sr_stats* st);

/* sr_generate_dev -- as sr_generate with DEVICE prompt and outputs, enqueued on `stream`;
 * the call returns after the outputs are written (it synchronises `stream`). */
sr_status sr_generate_dev(sr_ctx* ctx, const int32_t* prompt_dev, int P, int N, float alpha, const sr_schedule* sched,
                          int max_new, float temperature, float eos_bias, int eos_id, uint64_t seed,
                          int32_t* out_tokens_dev, int* out_len_dev, float* out_score_dev, sr_stats* st, void* stream);

/*
 * Component calls: Algorithm 1 one stage at a time on a batch object.
 * sr_batch_begin prefills the prompt through both models, admits candidates
 * 0..N-1 (shared prompt pages plus one private tail page each when P % 16 != 0)
 * and samples token 0 of every candidate.  The "round batch" is every
 * candidate that survived the previous round: live ones and those completed
 * since (Section 4.2: R_partial ranges over k = 1..b).
 */
sr_status sr_batch_begin(sr_ctx* ctx, const int32_t* prompt, int P, int N, int max_new, float temperature,
                         float eos_bias, int eos_id, uint64_t seed, sr_batch** out);
/* One decode step for every live candidate (Eq. auto-regressive): append the
 * last token's KV, run the generator, sample the next token.  logits_out (host,
 * nullable) receives the [b_live][vocab] fp32 logits in ascending candidate id.
 * SR_ERR_OOM if the pool cannot give each live candidate its page; SR_ERR_STATE
 * if no candidate is live. */
sr_status sr_decode_step(sr_ctx* ctx, sr_batch* batch, float* logits_out);
/* Partial rewards s(Y_k^{<=tau_k}) of the round batch (Eq. partial.reward.set),
 * tau_k = tokens generated so far.  rewards (host) gets b floats in ascending
 * candidate id; *b_out (nullable) gets b. */
sr_status sr_score_partial(sr_ctx* ctx, sr_batch* batch, float* rewards, int* b_out);
/* One rejection round on given partial rewards (host, b floats, ascending id):
 * r_cut = q_alpha(rewards) as the floor(alpha b)-th order statistic (Eq.
 * cutoff.threshold), I_accepted = {k : r_k >= r_cut} (Eq. accepted.set);
 * completed candidates join I with their reward; rejected live ones release
 * their pages; survivors are compacted.  Outputs: *r_cut_out, accepted ids
 * (host, ascending, capacity b), *b_out = |I_accepted| (accepted_ids_out and
 * b_out count completed candidates too), *b_live_out (nullable) = live after. */
sr_status sr_reject_compact(sr_ctx* ctx, sr_batch* batch, const float* rewards, float alpha, float* r_cut_out,
                            int32_t* accepted_ids_out, int* b_out, int* b_live_out);
/* Host snapshot of the batch state; any pointer may be NULL.
 *   ids_live [N], lengths [N], status [N] (0 live, 1 completed-unscored,
 *   2 completed-scored, 3 rejected), tokens [N][max_new], page_table [N][max_pages],
 *   free_stack [pool pages] (bottom first); counts: n_live, free_top, max_pages. */
sr_status sr_batch_query(sr_ctx* ctx, const sr_batch* batch, int32_t* ids_live, int32_t* lengths, int32_t* status,
                         int32_t* tokens, int32_t* page_table, int32_t* free_stack, int* n_live, int* free_top,
                         int* max_pages);
void sr_batch_end(sr_ctx* ctx, sr_batch* batch);

/*
 * Kernel-level entry points (device pointers, asynchronous on `stream`).
 * They run the same kernels as the calls above, for parity testing.
 */

/* Gumbel-max sampling (Eq. auto-regressive realised as in the Section 3
 * sampling step): token[r] = argmax_v (logits[r][v] + eos_bias [v == eos_id]) / T + g_v,
 * g_v = -ln(-ln u_v), u_v from Philox4x32-10 keyed (seed; v/4, orig_ids[r], steps[r], 0).
 * logits: fp32, row r at logits + r * ld (ld = 0 broadcasts one row).  b rows.
 * logprob_sum (device, nullable, indexed by orig_ids[r]): += ln softmax(logits[r])[token[r]] in
 * float64 (Section 5.3 self-likelihood; raw logits, NaN = -inf). */
sr_status sr_k_sample(const float* logits, long long ld, int b, int vocab, const int32_t* orig_ids,
                      const int32_t* steps, uint64_t seed, float temperature, float eos_bias, int eos_id,
                      int32_t* tokens_out, void* stream,
                      double* logprob_sum);

/* LM head fused with sampling (Section 3 sampling step, as sr_k_sample, without storing logits):
 * token[r] = the Gumbel-max sample of sr_k_sample over logits[r][v] = x[r] . W[v] (fp32 accumulation of
 * `dtype` operands, SR_DT_F16 or SR_DT_BF16), with step = lens[orig_ids[r]] as the token index of the noise.
 * x [M][K], W [vocab][K] (device, 16-byte aligned), K % 8 == 0, vocab % 32 == 0.  The GEMM's epilogue
 * reduces each row's 64-id chunks to a 32-byte record; a second kernel picks the token.  The token equals
 * sr_k_sample's on the logits sr_k_gemm (epilogue 0) computes with the same tile configuration: 256 x 256
 * CTA-pair tiles from 512 rows, 128 x 256 tiles below.  Allocates M * ceil(vocab / 64) * 32 bytes of
 * workspace on `stream` for the call. */
sr_status sr_k_lm_head_sample(int dtype, const void* x, const void* W, int M, int vocab, int K,
                              const int32_t* orig_ids, const int32_t* lens, uint64_t seed, float temperature,
                              float eos_bias, int eos_id, int32_t* tokens_out, void* stream);

/* r_cut selection (Eqs. cutoff.threshold, accepted.set) on b <= 4096 fp32
 * rewards: k = min(floor(alpha b), b - 1) (or k_override >= 0); r_cut = k-th
 * smallest by radix select on order-preserving keys; mask[i] = rewards[i] >= r_cut. */
sr_status sr_k_rcut(const float* rewards, int b, float alpha, int k_override, float* r_cut_out, uint8_t* mask_out,
                    void* stream);

/* Dense layer C = A W^T (fp32 accumulate).  dtype SR_DT_F16 or SR_DT_BF16 runs the
 * tcgen05 tensor-core kernel, SR_DT_F32 the fp32 SIMT kernel.  A [M][K] (lda = K),
 * W [N][K], both of `dtype`.  epilogue: 0 store fp32 C [M][N]; 1 add into fp32
 * C [M][N]; 2 store C as `dtype`; 3 SwiGLU / 4 GeGLU on column pairs
 * interleaved in blocks of 16 (W rows 32j..32j+15 gate block j, 32j+16..32j+31
 * up block j) storing `dtype` C [M][N/2]; 5 tanh-GELU storing `dtype` C [M][N]
 * (3-5 16-bit only).  Needs K % 8 == 0, N % 32 == 0 (N % 64 for 3, 4). */
sr_status sr_k_gemm(int dtype, const void* A, const void* W, void* C, int M, int N, int K, int epilogue,
                    void* stream);

/* Paged GQA decode attention for one layer: for slot s (candidate orig_ids[s])
 * and query head j, out[s][j] = softmax_t(q[s][j] . K_t / sqrt(dh)) V_t over
 * positions t in [max(0, len[s] - window), len[s]) read from the pool pages
 * page_table[orig_ids[s]][t / 16].  pool layout [page][2 (K,V)][n_kv][16][dh]
 * of `dtype` (pool points at this layer's page 0); q, out [b][n_heads][dh] `dtype`.
 * shared_pos (a multiple of 16, < every len; 0 = none): positions [0, shared_pos)
 * are in the same pages for every candidate (the shared prompt, Section 4.2's batch
 * of N responses to one prompt) and are read once per 64 candidates by a
 * tensor-core prefix pass (16-bit types only). */
sr_status sr_k_decode_attention(int dtype, const void* q, const void* pool, const int32_t* page_table, int pt_stride,
                                const int32_t* orig_ids, const int32_t* lens, int b, int n_heads, int n_kv_heads,
                                int head_dim, int window, int shared_pos, void* out, void* stream);

/* sr_k_decode_attention_static -- the same decode attention for callers that cannot allocate
 * device memory when they call (a server that has reserved all GPU memory up front, an
 * allocator-free embedding, a caller holding a lock an allocation could block on).  The paper has
 * no counterpart; this is an interface convenience.  Instead of a per-call buffer, the split
 * partials (needed when a context exceeds 512 positions) use one fixed 8 MiB device array that
 * every GPU loading the library holds until exit; the call allocates nothing.
 *   max_len : an upper bound on lens[]; it sizes the number of 512-position splits,
 *             ceil(min(max_len, window or max_len) / 512).  No shared-prefix pass (shared_pos = 0).
 * Rejects, with SR_ERR_INVALID_ARG and a message, shapes needing more than 2^21 scratch floats
 * (b * n_heads * splits * (head_dim + 2)).  lens[] is read on the device: a row whose length needs
 * more splits than max_len gives is computed over its first `splits` splits only (nothing is read
 * or written outside the array), a device flag records it, and the call returns SR_ERR_INVALID_ARG
 * with `out` not valid.  To read that flag the call synchronises `stream` before it returns.  The
 * first call on a device looks up the array's device address (cudaGetSymbolAddress) with that
 * device current; make that first call before any stream capture.  All calls share the array and
 * it keeps the last call's contents (every partial a call reads it has written itself, and the
 * flag is cleared at the start of each call); calls that overlap on the GPU, e.g. on two streams,
 * race on it. */
sr_status sr_k_decode_attention_static(int dtype, const void* q, const void* pool, const int32_t* page_table,
                                       int pt_stride, const int32_t* orig_ids, const int32_t* lens, int b,
                                       int n_heads, int n_kv_heads, int head_dim, int window, int max_len, void* out,
                                       void* stream);

/* Causal prefill attention over packed variable-length sequences with an
 * optional shared prefix.  Sequence j owns query/key rows seq_off[j] ..
 * seq_off[j+1]-1 of q [rows][n_heads][dh] and k, v [rows][n_kv][dh], at positions
 * pos0 + (row - seq_off[j]); every sequence also sees the n_pre prefix keys
 * k_pre, v_pre [n_pre][n_kv][dh] at positions 0..n_pre-1.  dtype SR_DT_F16 or SR_DT_BF16. */
sr_status sr_k_prefill_attention(int dtype, const void* q, const void* k, const void* v, const void* k_pre,
                                 const void* v_pre, int n_pre, const int32_t* seq_off, int n_seq, int pos0,
                                 int n_heads, int n_kv_heads, int head_dim, int window, void* out, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* SR_H */
