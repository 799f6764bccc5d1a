/*
 * tlf.h -- C ABI of the GB300 (sm_103a) decode-step library for T-LoopFormer,
 * a looped transformer with token-level elastic depth.
 *
 * The operation (T-LoopFormer, Sec. 3.2-3.3 and App. B):
 *   - a token-choice router maps each token's initial state h^(0) = E[x] to a
 *     loop count m in 1..M (Eq. 2-5);
 *   - loop i applies the shared J-layer block only to the tokens with m >= i,
 *     gathered into a dense list and scattered back (Eq. 6-7);
 *   - each (loop i, layer j) keeps its own KV cache; a token writes its k, v
 *     into cache (i, j) only when it runs loop i, and its loop-i query attends
 *     only to cache (i, j) (Eq. 8-11);
 *   - exited tokens keep h^(m), which goes through the final RMSNorm and the
 *     tied LM head.
 *
 * Block layout (the workloads' restatement of the paper's NanoGPT block):
 * pre-norm RMSNorm (eps from the config, gains stored), multi-head attention
 * with grouped kv heads and rotary position embedding at the token's original
 * position (pairs (k, k + head_dim/2), angle pos * rope_base^(-2k/head_dim)),
 * and a SwiGLU MLP; the router is RMSNorm (no gain) then a d -> M linear map
 * with bias. A decoding token appends its own entry to cache (i, j) and then
 * attends to every entry of it, itself included.
 *
 * Conventions for every call:
 *   - Return value: TLF_OK (0) or a negative TLF_ERR_* code; on error
 *     tlf_last_error(ctx) holds a one-line message. A call that fails changes
 *     no sequence state: validation and page reservation finish before any
 *     device work is queued.
 *   - Pointers marked "host" are ordinary CPU memory; pointers marked
 *     "host or device" are looked up with cudaPointerGetAttributes.
 *   - The caller owns every buffer it passes; the library copies what it keeps.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream). Calls that
 *     return loop counts synchronise that stream before returning.
 *   - Matrices are row-major with the output dimension first (y = W x).
 *     "dtype" means float32 when cfg.dtype == TLF_DTYPE_F32 and bfloat16 bit
 *     patterns (uint16) when cfg.dtype == TLF_DTYPE_BF16.
 *   - Not thread-safe: one thread drives a context at a time.
 */
#ifndef TLF_H_
#define TLF_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum tlf_status {
  TLF_OK = 0,
  TLF_ERR_INVALID_ARG = -1,   /* bad config, shape, pointer or duplicate id in a batch */
  TLF_ERR_UNKNOWN_SEQ = -2,   /* sequence id not live */
  TLF_ERR_DUPLICATE_SEQ = -3, /* sequence id already live */
  TLF_ERR_OUT_OF_PAGES = -4,  /* the KV page pool cannot hold the step */
  TLF_ERR_SEQ_TOO_LONG = -5,  /* sequence would exceed cfg.max_seq_len */
  TLF_ERR_CUDA = -6,          /* a CUDA runtime call failed */
  TLF_ERR_BAD_WEIGHTS = -7,   /* missing weight pointer */
  TLF_ERR_DEVICE = -8,        /* a kernel gave up a bounded wait or saw a bad index */
  TLF_ERR_NO_DEVICE = -9,     /* host-only context: the call needs a GPU */
  TLF_ERR_CAPACITY = -10      /* too many live sequences or batch larger than cfg.max_batch */
};

enum tlf_dtype { TLF_DTYPE_F32 = 0, TLF_DTYPE_BF16 = 1 };

/* Exit rule (Sec. 3.2). ARGMAX: m = 1 + argmax_l z_l, ties to the smaller
 * depth, margin = z_(1) - z_(2). SURVIVAL (Eq. 3-5): pi = softmax(z),
 * p^(i) = sum_{l>=i} pi_l, m = max{i : p^(i) > threshold}, margin =
 * min(p^(m) - threshold, threshold - p^(m+1)), p^(M+1) = 0. */
enum tlf_exit_rule { TLF_EXIT_ARGMAX = 0, TLF_EXIT_SURVIVAL = 1 };

/* GEMM implementation for bf16 models: AUTO = tcgen05/TMEM tensor-core
 * kernels; SIMT = CUDA-core kernels (the only choice for float32 models,
 * also used by tests as a second GPU path). */
enum tlf_gemm_impl { TLF_GEMM_AUTO = 0, TLF_GEMM_SIMT = 1 };

/* Ablations of the decode step (Sec. 4 ablation study, gather-scatter and
 * recursion-wise KV cache). Each computes the same logits and loop counts as
 * TLF_ABLATION_NONE and differs only in the work it does:
 *   NO_GATHER  every loop r that has an active token runs the shared block on
 *              all B rows of the step; rows with m <= r are masked: their
 *              residual stream is not updated and they append nothing, but
 *              their projections and attention over their loop-r caches run
 *              (the cost of computing without the gather of Eq. 6).
 *   DENSE_CACHE without recursion-wise caches: every loop's cache keeps a slot
 *              for every position (all M caches have the sequence's length);
 *              a token that exits before loop r leaves a masked slot there
 *              (position -1), and attention at loop r reads every slot and
 *              skips the masked ones (the mask mu^(r) of Eq. 10 applied to a
 *              full-length cache). bf16 models only; prefill runs position by
 *              position; tlf_cache_len counts slots and tlf_read_cache returns
 *              masked slots with position -1. */
enum tlf_ablation { TLF_ABLATION_NONE = 0, TLF_ABLATION_NO_GATHER = 1, TLF_ABLATION_DENSE_CACHE = 2 };

typedef struct tlf_config {
  int32_t vocab;        /* V; the LM head is tied to the embedding */
  int32_t d_model;      /* d, multiple of 64 */
  int32_t n_heads;      /* query heads Hq */
  int32_t n_kv_heads;   /* kv heads Hkv, divides Hq (grouped-query attention) */
  int32_t head_dim;     /* hd in {16, 32, 64, 128} */
  int32_t n_layers;     /* J layers in the shared block */
  int32_t ffn_hidden;   /* SwiGLU hidden width, multiple of 16 */
  int32_t max_loops;    /* M (user-set maximum depth, Sec. 3.2), 1..16 */
  float rope_base;      /* 10000 */
  float norm_eps;       /* RMSNorm eps, 1e-5 */
  int32_t dtype;        /* tlf_dtype: weights, activations between kernels and KV pages */
  int32_t exit_rule;    /* tlf_exit_rule */
  float threshold;      /* survival threshold (Eq. 4), 0.5 */
  int32_t max_seqs;     /* live sequences held at once */
  int32_t max_batch;    /* tokens per decode step, 1..256 */
  int32_t max_seq_len;  /* tokens per sequence */
  int32_t page_size;    /* tokens per KV page, multiple of 16 (64 is a good default) */
  int32_t gemm_impl;    /* tlf_gemm_impl */
  int32_t host_only;    /* 1: allocate nothing on a GPU; only validation and bookkeeping run */
  int32_t prefill_chunk;/* prompt tokens per batched-prefill chunk (bf16 models); 0 = 8192 */
  int64_t kv_pool_pages;/* pages in the KV pool; 0 = max_seqs * max_loops * ceil(max_seq_len / page_size) */
  int32_t ablation;     /* tlf_ablation; 0 = the method as published */
  int32_t conditioning; /* 0 = none (the workloads' backbone); 1 = time/step AdaLN conditioning
                         * (Sec. 3.1, App. A), with the cond_* and mod_* weights: a token of depth m
                         * runs loop i conditioned on t = (i-1)/m and Delta = 1/m; layer j computes
                         * x += alpha_msa * MHSA(RMSNorm(x) * g * (1 + gamma_msa)) and
                         * x += alpha_mlp * FFN(RMSNorm(x) * g * (1 + gamma_mlp)) */
  int32_t router_hidden;/* 0 = linear router d -> M (the workloads); H_r > 0 (multiple of 8, <= 8192) = the
                         * two-layer MLP router of Sec. 3.2: z = W_r GELU(W_1 RMSNorm(h0) + b_1) + b_r
                         * with the exact GELU, weights router_w1/router_b1, router_w then [M][H_r] */
  int32_t reserved;     /* must be 0 */
} tlf_config;

/* Host pointers to the weights. Shapes use V, d, Hq, Hkv, hd, J, ff, M from
 * the config. Norm gains and the router bias are float32; every other matrix
 * is in the config dtype. The library copies them to the GPU in tlf_create. */
typedef struct tlf_weights {
  const void* embedding;   /* [V][d] */
  const void* router_w;    /* [M][d], or [M][H_r] with the MLP router */
  const float* router_b;   /* [M] */
  const void* wq;          /* [J][Hq*hd][d] */
  const void* wk;          /* [J][Hkv*hd][d] */
  const void* wv;          /* [J][Hkv*hd][d] */
  const void* wo;          /* [J][d][Hq*hd] */
  const void* w_gate;      /* [J][ff][d] */
  const void* w_up;        /* [J][ff][d] */
  const void* w_down;      /* [J][d][ff] */
  const float* attn_norm;  /* [J][d] */
  const float* mlp_norm;   /* [J][d] */
  const float* final_norm; /* [d] */
  /* Time/step conditioning (cfg.conditioning = 1; may be NULL otherwise), float32. For each of the
   * scalars t and Delta: 256 sinusoidal features [cos(x w_1), sin(x w_1), ...], w_k =
   * 10000^(-(k-1)/128), then w2 SiLU(w1 f + b1) + b2; c = sum of the two; layer j's modulator
   * gives mod_w[j] SiLU(c) + mod_b[j] = (alpha_msa, alpha_mlp, gamma_msa, gamma_mlp), d each. */
  const float* cond_t_w1;  /* [d][256] */
  const float* cond_t_b1;  /* [d] */
  const float* cond_t_w2;  /* [d][d] */
  const float* cond_t_b2;  /* [d] */
  const float* cond_dt_w1; /* [d][256] */
  const float* cond_dt_b1; /* [d] */
  const float* cond_dt_w2; /* [d][d] */
  const float* cond_dt_b2; /* [d] */
  const float* mod_w;      /* [J][4d][d] */
  const float* mod_b;      /* [J][4d] */
  const void* router_w1;   /* [H_r][d] (cfg.router_hidden > 0; may be NULL otherwise) */
  const float* router_b1;  /* [H_r] */
} tlf_weights;

typedef struct tlf_ctx tlf_ctx;

/* Validate a configuration without touching a GPU. Returns TLF_OK or
 * TLF_ERR_INVALID_ARG; `msg` (may be NULL) receives a NUL-terminated reason. */
int tlf_validate_config(const tlf_config* cfg, char* msg, size_t msg_len);

/* Bytes of one KV page: n_layers * 2 (K, V) * n_kv_heads * page_size *
 * head_dim * element size. Pages are shared by the J layers of one
 * (sequence, loop) cache. Returns 0 for an invalid config. */
int64_t tlf_page_bytes(const tlf_config* cfg);

/* Create a context (Sec. 3.2-3.3): validate cfg, copy the weights of the
 * shared J-layer block, the router and the tied embedding to the current CUDA
 * device, and allocate the KV page pool that holds the recursion-wise caches
 * of Sec. 3.3 (Eq. 8: one cache per loop i <= M, the user-set maximum depth
 * of Sec. 3.2, and per layer j) plus the step workspaces. Weights are copied;
 * the caller keeps ownership of w. *out receives the context (NULL on
 * failure). On failure the message is available through tlf_last_error(NULL)
 * on the same thread. Errors: INVALID_ARG (cfg), BAD_WEIGHTS (a required
 * pointer is NULL), CUDA (no sm_103a device, allocation failure).
 *
 * Environment switches select equivalent comparison paths, each covered by
 * the GPU tests. The first two change only how kernels are launched, and the
 * results are bit-identical; the others change rounding, within the logits
 * tolerance.
 *   TLF_NO_GRAPH=1       launch each step's kernels directly instead of
 *                        replaying a captured CUDA graph (read here)
 *   TLF_NO_PDL=1         plain stream order instead of programmatic
 *                        dependent launch (read when the library loads)
 *   TLF_NO_SPLIT_NORM=1  every decode pre-norm as a kernel of its own instead
 *                        of split across the neighbouring GEMMs (read here)
 *   TLF_NO_OPERAND_LO=1  one bf16 plane for the decode GEMMs' activation
 *                        operands instead of hi + lo (two-term) planes (read
 *                        here)
 *   TLF_PF_ATTN_V1=1     prefill attention with every thread staging and
 *                        re-laying out each K/V page instead of the
 *                        warp-specialised kernel that loads pages with a
 *                        tensor map (read here; same arithmetic, different
 *                        rounding order of the row sums) */
int tlf_create(const tlf_config* cfg, const tlf_weights* w, tlf_ctx** out);

/* Free every device and host resource of the context: the weights, the
 * page pool with every sequence's recursion-wise caches (Sec. 3.3, Eq. 8) and
 * the workspaces. Live sequences end with it. NULL is a no-op. Synchronises
 * the device before freeing, so no queued step reads freed memory. */
void tlf_destroy(tlf_ctx* ctx);

/* Message of the last failed call on ctx (or of the last failed tlf_create
 * on this thread when ctx is NULL). Never NULL. */
const char* tlf_last_error(const tlf_ctx* ctx);

/* Prefill (Sec. 3.3, "prefill" in App. B): create n_seqs new sequences and
 * run their prompts. Prompt s is tokens[offsets[s] .. offsets[s+1]) (host,
 * offsets has n_seqs+1 entries, every prompt non-empty). Each prompt token is
 * routed, and runs its loops in position order; its k, v land in the caches
 * of the loops it runs, at its original position.
 *   seq_ids      host [n_seqs], distinct, not live
 *   forced       host [offsets[n_seqs]] or NULL; entries >= 1 replace the
 *                router's loop count (fixed-depth runs), others are ignored
 *   last_logits  host or device float32 [n_seqs][V] or NULL: logits after
 *                each prompt's last token
 *   loops        host int32 [offsets[n_seqs]] or NULL: loop count per token
 * The prompts run in chunks of at most prefill_chunk tokens; the call
 * synchronises `stream` within every chunk (the rows of each loop of a chunk
 * of more than 256 tokens come to the host to size that loop's launches, and
 * the loop counts at its end) and before returning.
 * Errors: INVALID_ARG, DUPLICATE_SEQ, CAPACITY, SEQ_TOO_LONG, OUT_OF_PAGES,
 * CUDA, DEVICE. */
int tlf_prefill(tlf_ctx* ctx, int32_t n_seqs, const uint64_t* seq_ids, const int32_t* offsets,
                const int32_t* tokens, const int32_t* forced, float* last_logits, int32_t* loops,
                void* stream);

/* One decode step (Sec. 3.3, Eq. 9-11): one new token for each of `batch`
 * live, distinct sequences. The router picks each token's loop count; loop i
 * runs on the dense list of tokens with m >= i; each token appends k, v to
 * the loop-i caches of its sequence and attends to them.
 *   seq_ids        host [batch]
 *   tokens         host [batch] token ids in [0, V)
 *   forced         host [batch] or NULL; entries >= 1 replace the router's
 *                  loop count
 *   logits         host or device float32 [batch][V]; NULL skips the LM head
 *   loops          host int32 [batch] (required): the loop counts m
 *   router_margin  host float32 [batch] or NULL: the router's decision margin
 *                  (see tlf_exit_rule); a token is a near-tie when it is small
 * The call synchronises `stream` before returning (loop counts are host
 * outputs). Errors: INVALID_ARG, UNKNOWN_SEQ, CAPACITY, SEQ_TOO_LONG,
 * OUT_OF_PAGES, CUDA, DEVICE. */
int tlf_decode_step(tlf_ctx* ctx, int32_t batch, const uint64_t* seq_ids, const int32_t* tokens,
                    const int32_t* forced, float* logits, int32_t* loops, float* router_margin,
                    void* stream);

/* End a sequence: return the pages of its M recursion-wise caches (Sec. 3.3,
 * Eq. 8: the loop-i caches of every layer j) to the pool and free its slot.
 * The id may be reused by a later tlf_prefill or tlf_load_cache. Host-side
 * only: queues no device work. Errors: UNKNOWN_SEQ. */
int tlf_release(tlf_ctx* ctx, uint64_t seq_id);

/* Create a sequence whose recursion-wise caches hold a given snapshot (a
 * restored session). For loop i (0-based), lens[i] entries at original
 * positions positions[off_i .. off_i + lens[i]) with off_i = sum_{i'<i}
 * lens[i'], strictly increasing; loop 0 must hold 0..lens[0]-1, and each
 * loop's positions must be a subset of the previous loop's (active sets
 * nest, Eq. 4-5). k and v are host arrays in the config dtype laid out
 * [sum lens][J][Hkv][hd] in the same loop order, already rotated (RoPE at
 * their positions). The next token of the sequence has position lens[0].
 * With k = v = NULL the entries are filled on the device instead, element x
 * of the pool getting (fmix32(x) mod 256 - 128) / 64 (fmix32 = the 32-bit
 * MurmurHash3 finaliser): for long caches whose values do not matter, such
 * as throughput runs.
 * Errors: INVALID_ARG, DUPLICATE_SEQ, CAPACITY, SEQ_TOO_LONG, OUT_OF_PAGES,
 * CUDA, NO_DEVICE. */
int tlf_load_cache(tlf_ctx* ctx, uint64_t seq_id, const int32_t* lens, const int32_t* positions,
                   const void* k, const void* v);

/* ---- kernel-level operation: recursion-wise decode attention ------------- */

/* One query per row against that row's KV cache (Eq. 10 on a cache that
 * holds only valid entries, so no mask is needed): for row b and query head
 * h, out[b][h] = softmax(q[b][h] . K_b^T / sqrt(hd)) V_b over the first
 * lens[b] entries of the cache addressed by page_table[b], kv head
 * h / (n_heads / n_kv_heads). The same split-K kernels serve tlf_decode_step.
 * All pointers are device pointers. Page layout, in the dtype:
 * [n_pages][n_layers][2 (K, V)][n_kv_heads][page_size][head_dim]; entry e of
 * row b sits in page page_table[b * max_pages + e / page_size] at offset
 * e % page_size. */
typedef struct tlf_attn_args {
  int32_t n;            /* rows (queries), 1..256 */
  int32_t n_heads;      /* Hq */
  int32_t n_kv_heads;   /* Hkv, divides Hq */
  int32_t head_dim;     /* hd (same choices as tlf_config) */
  int32_t n_layers;     /* layers stored per page */
  int32_t layer;        /* layer whose K/V are read, 0..n_layers-1 */
  int32_t page_size;    /* 64 */
  int32_t dtype;        /* tlf_dtype of the pool and of out */
  int32_t max_pages;    /* entries per page-table row */
  int32_t reserved0;
  int64_t n_pages;      /* pages in the pool (page ids are checked against it) */
  const float* q;       /* [n][Hq][hd] float32, already rotated */
  const void* pool;     /* KV pages */
  const int32_t* page_table; /* [n][max_pages] */
  const int32_t* lens;  /* [n] keys per row, 1..max_pages*page_size */
  void* out;            /* [n][Hq*hd] in the dtype */
  uint32_t* err;        /* optional device word: bit 1 = a bounded wait expired, bit 2 = bad page id */
} tlf_attn_args;

/* Scratch bytes tlf_attn_decode needs for these arguments on the current
 * device (split-K work plan and partial results); 0 for invalid arguments. */
size_t tlf_attn_decode_scratch_bytes(const tlf_attn_args* a);

/* Launch the attention on `stream` (cudaStream_t) using caller-provided
 * device scratch of at least tlf_attn_decode_scratch_bytes(a) bytes. Does not
 * synchronise. Errors (INVALID_ARG, CUDA) are reported through
 * tlf_last_error(NULL) on the calling thread. */
int tlf_attn_decode(const tlf_attn_args* a, void* scratch, size_t scratch_bytes, void* stream);

/* The same attention as tlf_attn_decode, for callers that cannot allocate
 * device memory: for instance a plug-in whose host application owns every
 * byte of the GPU through its own pool, or a request path where a
 * cudaMalloc (which can synchronise the device and stall other work) is not
 * allowed. It allocates nothing; its scratch is a 4 MiB array built into the
 * library, present on every GPU that loads the library until the process
 * exits. Arguments whose scratch (tlf_attn_decode_scratch_bytes) exceeds
 * 4 MiB are rejected with TLF_ERR_INVALID_ARG and a message naming the
 * sizes; a C4-shaped call (16 rows, Hq 16 / Hkv 8, hd 128) needs under 1
 * MiB. The first call on a device looks up the array's device address (a
 * set-up step), so make that first call before any stream capture. The
 * address is remembered per device and per CUDA context: after the context
 * is destroyed and re-created (cudaDeviceReset, for one) the next call looks
 * it up again, so make that call, too, before any stream capture. Every
 * call on a device shares the array and it keeps the last call's contents:
 * calls whose kernels overlap on the GPU (different streams, or other host
 * threads) race and must not be issued; serialise them. Launches on
 * `stream` without synchronising; errors as for tlf_attn_decode. The paper
 * has no counterpart of this entry point. */
int tlf_attn_decode_static(const tlf_attn_args* a, void* stream);

/* ---- inspection ---------------------------------------------------------- */

/* Number of live sequences and free pages. */
int tlf_stats(const tlf_ctx* ctx, int32_t* live_seqs, int64_t* free_pages, int64_t* total_pages);

/* Entries in the loop-`loop` caches (1-based loop) of a sequence; all J layers share it. */
int tlf_cache_len(const tlf_ctx* ctx, uint64_t seq_id, int32_t loop, int32_t* len);

/* Copy cache (loop, layer) of a sequence to the host: positions int32 [len],
 * k and v float32 [len][Hkv][hd] (widened from the storage dtype). `loop` is
 * 1-based, `layer` 0-based. Any output pointer may be NULL. */
int tlf_read_cache(tlf_ctx* ctx, uint64_t seq_id, int32_t loop, int32_t layer, int32_t* positions,
                   float* k, float* v);

/* Active sets of the last decode step (Eq. 4-6): counts[i] = |A_{i+1}| for
 * i < M, and idx[i * batch + r] for r < counts[i] the batch rows of A_{i+1}
 * in increasing order. Host arrays [M] and [M * batch]. */
int tlf_last_active_sets(tlf_ctx* ctx, int32_t* counts, int32_t* idx);

/* Kernel-level timing of the last decode step, filled when
 * tlf_set_profiling(ctx, 1) is on: milliseconds spent in the recursion-wise
 * attention kernels, the KV bytes they read (K and V of every visited entry
 * once per kv head), and the number of kernels launched. */
int tlf_set_profiling(tlf_ctx* ctx, int32_t on);
int tlf_last_step_profile(const tlf_ctx* ctx, float* attn_ms, double* attn_kv_bytes,
                          int32_t* kernel_launches);

/* Per-kernel-class milliseconds of the last decode step run with profiling
 * on (events between launches, so kernels do not overlap while profiled).
 * Classes, in order: 0 router, 1 plan (compaction), 2 attention pre-norm,
 * 3 QKV GEMM, 4 RoPE + append, 5 attention, 6 O GEMM + residual, 7 MLP
 * pre-norm, 8 gate/up GEMM, 9 SwiGLU, 10 down GEMM + residual, 11 final
 * norm, 12 LM head. Writes min(n, 13) entries of ms; returns TLF_OK. */
int tlf_last_step_kernel_times(const tlf_ctx* ctx, float* ms, int32_t n);

#ifdef __cplusplus
}
#endif
#endif /* TLF_H_ */
