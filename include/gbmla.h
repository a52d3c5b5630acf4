/*
 * gbmla.h -- C ABI of libgbmla.so: the absorbed multi-head latent attention
 * (MLA) decode step of a converted MLA draft model, on one GB300 (sm_103a).
 *
 * The step a draft runs at every proposal (q_len = 1) and every catch-up
 * chunk (q_len = gamma + 1) is
 *
 *   mla_project_append (optional, replaces mla_cache_append when the caller
 *                      holds hidden states) project h into the latent and
 *                      positional caches and the queries     (Sec. 3.2, Eq. 1)
 *   mla_cache_append   write this step's latent rows c_j and RoPE-rotated
 *                      positional keys k_j^PE into the cache    (Sec. 3.2, Sec. 3.1)
 *   mla_absorb_q       q_lat = W_UK[g]^T q_nope, RoPE the positional query
 *                      (attention "through absorbed projections", Sec. 1;
 *                      the algebra is Eq. 5 read right to left)
 *   mla_decode_attn    split-KV attention over the latent cache: scores
 *                      q_lat . c_j + q_rot . k_j^PE under one scale, causal
 *                      softmax, o_lat = sum_j a_j c_j          (Eqs. 2-4, Sec. 3.3)
 *   mla_combine        merge the per-split partials with their log-sum-exp
 *                      (the softmax normaliser of Eq. 3)
 *   mla_out_proj       o = W_UV[g] o_lat, optionally out = W_O concat_h o
 *                      (Eq. 5; the block output "after its fixed output
 *                      projection", Sec. 4.1)
 *
 * mla_decode_step runs append (optional), absorption, attention, combine and
 * the projections in one call.
 *
 * Conventions shared by every entry point
 *   - All pointers except the two structs are DEVICE pointers on the current
 *     CUDA device.  The caller owns and allocates every buffer; the library
 *     allocates no memory on any call.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Every call only enqueues work on it and returns; nothing
 *     synchronises except mla_check_status().
 *   - bf16 = IEEE bfloat16 stored as 2 bytes; all accumulation is fp32.
 *   - Row-major dense layouts; "[a, b, c]" lists dimensions outermost first.
 *   - Head h belongs to KV group g(h) = h / (H / G) (MHA is G = H, Sec. 3.1).
 *   - kv_len[b] is the number of cached tokens of sequence b AFTER this
 *     step's append.  Query i (0 <= i < q_len) of sequence b sits at position
 *     kv_len[b] - q_len + i and attends to keys 0 .. kv_len[b] - q_len + i
 *     (causal inside the chunk).  1 <= q_len <= 16 and q_len <= kv_len[b].
 *   - RoPE (Sec. 3.1, R_t): theta_k = rope_base^(-2k/d_rope); rope_style 0
 *     rotates the pair (k, k + d_rope/2), style 1 the pair (2k, 2k + 1).
 *     The positional cache stores keys already rotated to their position.
 *
 * Errors
 *   Host-side argument checks run before anything is enqueued and return
 *   MLA_ERR_INVALID_ARG or MLA_ERR_UNSUPPORTED; nothing was launched then.
 *   A failed launch returns MLA_ERR_CUDA.  Faults a kernel can only see on
 *   the device (a block-table entry outside [0, num_pages), a position past
 *   `capacity`, kv_len[b] < q_len, a bounded wait that ran out) never trap:
 *   the kernel records the fault in a sticky per-device status word, skips
 *   the offending work and returns.  mla_check_status() reports and clears
 *   it.  Outputs of a call that recorded a device fault are unspecified.
 */
#ifndef GBMLA_H
#define GBMLA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum mla_status {
    MLA_OK = 0,
    MLA_ERR_INVALID_ARG = 1,    /* a host-checked argument is wrong            */
    MLA_ERR_UNSUPPORTED = 2,    /* valid, but a size this build does not run   */
    MLA_ERR_CUDA = 3,           /* a CUDA runtime call or launch failed        */
    MLA_ERR_DEVICE_BOUNDS = 4,  /* device saw a bad page, position or length   */
    MLA_ERR_DEVICE_TIMEOUT = 5  /* a bounded device-side wait ran out          */
} mla_status;

/* Shape of one MLA layer (Sec. 3.1-3.2 notation). */
typedef struct mla_dims {
    int32_t num_heads;      /* H: query heads                                     */
    int32_t num_kv_groups;  /* G: KV groups of the source GQA model, H % G == 0   */
    int32_t d_nope;         /* non-positional query/key width per head            */
    int32_t d_rope;         /* decoupled positional key width (32 or 64)          */
    int32_t d_v;            /* value width per head                               */
    int32_t rank;           /* r: latent rank (128, 256 or 512)                   */
    int32_t hidden;         /* D: model width for W_O; 0 = no output projection   */
    float sm_scale;         /* softmax scale, 1/sqrt(d_k) of the converted head   */
    int32_t rope_style;     /* 0 rotate-half pairs, 1 interleaved pairs           */
    float rope_base;        /* RoPE base (e.g. 10000)                             */
} mla_dims;

/* The latent cache c [.., r] and the rotated positional-key cache
 * k_rope [.., d_rope] (Sec. 3.2), both bf16.  Token t of sequence b lives in
 * block blk at slot s:
 *   contiguous (block_table == NULL): blk = b,                               s = t
 *   paged      (block_table != NULL): blk = block_table[b*bt_stride + t/page_size],
 *                                     s = t % page_size
 * and its rows start at c_kv + blk*c_blk_stride + s*c_tok_stride and
 * k_rope + blk*r_blk_stride + s*r_tok_stride (strides in elements).
 * Requirements: both base pointers 16-byte aligned; all four strides
 * multiples of 8 elements; tok strides >= rank / d_rope; page_size == 64 when
 * paged.  The two caches may interleave (one [.., r + d_rope] row per token)
 * through the strides. */
typedef struct mla_cache {
    void *c_kv;
    void *k_rope;
    int64_t c_tok_stride, r_tok_stride;
    int64_t c_blk_stride, r_blk_stride;
    const int32_t *block_table;   /* device int32, NULL = contiguous     */
    int32_t bt_stride;            /* entries per block-table row         */
    int32_t page_size;            /* tokens per page (64) when paged     */
    int32_t num_pages;            /* pages in the pool when paged        */
    int32_t capacity;             /* most tokens one sequence may hold   */
} mla_cache;

/* Split-KV partitioning used by mla_decode_attn and mla_combine.  Each
 * sequence is cut into MLA_SPLIT_TILE-token tiles; the tiles of all
 * sequences, in batch order, form one list of T tiles, and partition k
 * (0 <= k < S) takes tiles [floor(k*T/S), floor((k+1)*T/S)).  A partition
 * writes one partial per sequence it touches, in slot b + k of o_part and
 * lse_part, so B + S - 1 slots always suffice. */
#define MLA_SPLIT_TILE 128

/* Sizes of the two partial buffers mla_decode_attn writes for this problem,
 * and the number of partitions S it will use: num_splits > 0 is taken as
 * given, 0 picks S from the device's SM count (the same rule every call of
 * this library applies): one partition per SM (per group of SMs sharing a
 * tile); when that leaves at most four tiles per partition (the tiles counted
 * as batch x ceil(max_kv_len / MLA_SPLIT_TILE)), the fewest partitions that
 * keep the same most tiles per partition.
 * max_kv_len bounds every kv_len[b].  Any output pointer may be NULL. */
mla_status mla_workspace_size(const mla_dims *dims, int32_t batch, int32_t q_len, int32_t max_kv_len,
                              int32_t num_splits, size_t *o_part_bytes, size_t *lse_part_bytes,
                              int32_t *num_splits_used);

/* Cache append (Sec. 3.2 latent cache c_j = W^DKV h_j and positional key
 * k^PE_j; Sec. 3.1 rotation).  For every sequence b and entry k < n_new,
 * position p = start_pos[b] + k:
 *   c_kv row (b, p)   <- c_new[b, k, :]                (bit-exact copy)
 *   k_rope row (b, p) <- bf16(R_p kr_new[b, k, :])     (fp32 rotation, RNE)
 *   c_new [batch, n_new, rank] bf16, kr_new [batch, n_new, d_rope] bf16
 *   (not yet rotated), start_pos [batch] int32 device.
 * A position outside [0, capacity) or a page outside [0, num_pages) is
 * skipped and recorded as MLA_ERR_DEVICE_BOUNDS.  batch or n_new == 0: no-op. */
mla_status mla_cache_append(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t n_new,
                            const void *c_new, const void *kr_new, const int32_t *start_pos, void *stream);

/* Projection of this step's hidden states into the cache and the queries,
 * the work that precedes mla_cache_append / mla_absorb_q, as one launch
 * (Sec. 3.2: latent c_j = W^DKV h_j and positional key k^PE_j = R_j W^KR h_j,
 * one key shared by all heads; Sec. 3.1 Eq. 1: q_{t,i} = W^Q_i h_t, whose
 * first d_nope entries take the non-positional path and the last d_rope the
 * rotary path).  For every sequence b and entry k < n_new, position
 * p = start_pos[b] + k and x = h[b, k, :]:
 *   c_kv row (b, p)     <- bf16(W_DKV x)          (fp32 accumulation, one RNE rounding)
 *   k_rope row (b, p)   <- bf16(R_p (W_KR x))     (the fp32 sum rotated in fp32, one rounding)
 *   q_nope[b, k, h, :]  <- bf16((W_Q x)[h dq .. h dq + d_nope))
 *   q_pe[b, k, h, :]    <- bf16((W_Q x)[h dq + d_nope .. (h + 1) dq))   (not rotated)
 * with dq = d_nope + d_rope.  h [batch, n_new, hidden] bf16 with
 * hidden = dims->hidden > 0 and a multiple of 8; W_DKV [rank, hidden],
 * W_KR [d_rope, hidden], W_Q [H dq, hidden] bf16; q_nope [batch, n_new, H,
 * d_nope] and q_pe [batch, n_new, H, d_rope] bf16; start_pos [batch] int32
 * device; every bf16 pointer 16-byte aligned.  w_q == NULL skips the queries
 * (q_nope and q_pe may then be NULL).  A position outside [0, capacity) or a
 * page outside [0, num_pages) skips that entry's cache rows and is recorded
 * as MLA_ERR_DEVICE_BOUNDS; its queries are still written.  batch or
 * n_new == 0: no-op. */
mla_status mla_project_append(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t n_new,
                              const void *h, const void *w_dkv, const void *w_kr, const void *w_q,
                              const int32_t *start_pos, void *q_nope, void *q_pe, void *stream);

/* Query absorption (Sec. 1; Eq. 5): for each (b, i, h)
 *   q_abs[b, i, h, 0:r]        = sum_d q_nope[b, i, h, d] * W_UK[g(h), d, :]
 *   q_abs[b, i, h, r:r+d_rope] = R_p q_pe[b, i, h, :],  p = kv_len[b] - q_len + i
 *   q_nope [batch, q_len, H, d_nope] bf16, q_pe [batch, q_len, H, d_rope] bf16,
 *   W_UK [G, d_nope, rank] bf16, kv_len [batch] int32 device,
 *   q_abs [batch, q_len, H, rank + d_rope] bf16 (output, unscaled). */
mla_status mla_absorb_q(const mla_dims *dims, int32_t batch, int32_t q_len, const void *q_nope,
                        const void *q_pe, const int32_t *kv_len, const void *w_uk, void *q_abs,
                        void *stream);

/* Split-KV attention core over the shared latent cache (Eqs. 2-4 with the
 * Sec. 3.3 score routing).  Every partition k reads each cache tile it owns
 * once for all heads and query positions and, for every sequence b it
 * touches, writes
 *   o_part[b + k, i, h, :]  = sum_j a~_j c_j / sum_j a~_j     (fp32, [.., rank])
 *   lse_part[b + k, i, h]   = ln sum_j exp(s_j)                (fp32, natural log)
 * over its own keys j, where s_j = sm_scale * (q_abs_lat . c_j + q_abs_rot . k_rope_j)
 * and a~_j = exp(s_j).  A query with no visible key in the partition gets
 * lse = -inf and o = 0.  P = softmax weights are rounded to bf16 before they
 * multiply the bf16 cache; everything else is fp32.
 *   q_abs [batch, q_len, H, rank + d_rope] bf16 (from mla_absorb_q),
 *   kv_len [batch] int32 device, max_kv_len >= every kv_len[b],
 *   o_part / lse_part sized by mla_workspace_size for the same arguments. */
mla_status mla_decode_attn(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t q_len,
                           const int32_t *kv_len, int32_t max_kv_len, const void *q_abs,
                           int32_t num_splits, float *o_part, float *lse_part, void *stream);

/* Merge the partials of each sequence (softmax normaliser of Eq. 3):
 *   M = max_k lse_k,  w_k = exp(lse_k - M),
 *   o_lat[b, i, h, :] = sum_k w_k o_part_k / sum_k w_k,  lse[b, i, h] = M + ln sum_k w_k
 * num_splits must resolve to the same S as in mla_decode_attn (pass the same
 * value, or the one mla_workspace_size returned).
 *   o_lat [batch, q_len, H, rank] fp32; lse [batch, q_len, H] fp32 or NULL. */
mla_status mla_combine(const mla_dims *dims, int32_t batch, int32_t q_len, int32_t num_splits,
                       const int32_t *kv_len, int32_t max_kv_len, const float *o_part,
                       const float *lse_part, float *o_lat, float *lse, void *stream);

/* Up-projection (Eq. 5) and output projection (Sec. 4.1):
 *   o[b, i, h, :]  = W_UV[g(h)] o_lat[b, i, h, :]            -> bf16 [batch, q_len, H, d_v]
 *   out[b, i, :]   = W_O concat_h o[b, i, h, :]               -> bf16 [batch, q_len, hidden]
 * (concat index h*d_v + e).  W_UV [G, d_v, rank] bf16, W_O [hidden, H*d_v]
 * bf16.  o is always written (W_O reads it, rounded to bf16); w_o == NULL or
 * hidden == 0 skips the second product and out may then be NULL. */
mla_status mla_out_proj(const mla_dims *dims, int32_t batch, int32_t q_len, const float *o_lat,
                        const void *w_uv, const void *w_o, void *o, void *out, void *stream);

/* One decode step in one call: mla_cache_append (of q_len new entries per
 * sequence at start_pos, when c_new is not NULL), mla_absorb_q,
 * mla_decode_attn, mla_combine and mla_out_proj, launched in that order on
 * `stream` with the arguments and buffers those five calls take (o_part and
 * lse_part sized by mla_workspace_size for the same batch, q_len, max_kv_len
 * and num_splits).  Every stage's arguments are checked before the first
 * launch: an error returns with nothing launched.  The results are those of
 * the five calls, bit for bit; one call instead of five saves the caller's
 * per-call overhead on short steps.  The paper has no counterpart (it is the
 * step of Sec. 3.2-3.3 as a whole). */
mla_status mla_decode_step(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t q_len,
                           const void *c_new, const void *kr_new, const int32_t *start_pos, const void *q_nope,
                           const void *q_pe, const int32_t *kv_len, int32_t max_kv_len, const void *w_uk,
                           const void *w_uv, const void *w_o, int32_t num_splits, void *q_abs, float *o_part,
                           float *lse_part, float *o_lat, float *lse, void *o, void *out, void *stream);

/* Acceptance statistics of a draft against its target at the same contexts
 * (Sec. 3.3), one row per context over a vocabulary of `vocab` tokens:
 *   p_D = softmax(draft row), p_T = softmax(target row)        (temperature 1)
 *   alpha_sample[r]  = sum_y min(p_D(y), p_T(y))                (Eq. 9, = 1 - TV)
 *   argmax_draft[r], argmax_target[r] = index of the largest logit, the lowest
 *                      index among equal maxima (decided on the logits)
 *   greedy_accept[r] = argmax_draft[r] == argmax_target[r]      (Eq. 10)
 * draft_logits / target_logits [rows, row_stride] (the first `vocab` entries of
 * each row used), fp32 (logits_dtype 0) or bf16 (1); both 16-byte aligned,
 * row_stride >= vocab and row_stride * element size a multiple of 16 bytes.
 * All arithmetic fp32.  Outputs [rows] device arrays; any may be NULL.
 * rows == 0: no-op.  The paper has no kernel for this; it reports the two
 * quantities its Eqs. 9-10 define. */
mla_status mla_acceptance_stats(int32_t rows, int32_t vocab, int32_t logits_dtype, const void *draft_logits,
                                const void *target_logits, int64_t row_stride, float *alpha_sample,
                                int32_t *argmax_draft, int32_t *argmax_target, int32_t *greedy_accept,
                                void *stream);

/* ---- The original GQA draft at the same shapes (Sec. 3.1, Eqs. 1-4): the
 * model the converted MLA draft replaces, for comparing cache bytes and step
 * time.  Each KV group g of sequence b has its own key and value cache; unit
 * u = b*G + g addresses them through an mla_cache whose k_rope holds the keys
 * (stored rotated to their position, head_dim per token) and c_kv the values
 * (head_dim per token), block u (contiguous) or block-table row u (paged),
 * with the same stride, alignment and page rules as the MLA cache. */
typedef struct mla_gqa_dims {
    int32_t num_heads;      /* H                                        */
    int32_t num_kv_groups;  /* G, H % G == 0                            */
    int32_t head_dim;       /* key = value width per head: 64 or 128    */
    float sm_scale;         /* 1/sqrt(head_dim)                         */
    int32_t rope_style;     /* as in mla_dims, over the whole head      */
    float rope_base;
} mla_gqa_dims;

/* New keys and values of every (sequence, group) at positions start_pos[b] + k:
 * keys rotated in fp32 and rounded once to bf16, values copied.
 *   k_new, v_new [batch, n_new, G, head_dim] bf16; start_pos [batch] int32.
 * Faults as for mla_cache_append. */
mla_status mla_gqa_append(const mla_gqa_dims *dims, const mla_cache *cache, int32_t batch, int32_t n_new,
                          const void *k_new, const void *v_new, const int32_t *start_pos, void *stream);

/* Partial-buffer sizes and split count of mla_gqa_decode_attn (as
 * mla_workspace_size, over the batch*G units). */
mla_status mla_gqa_workspace_size(const mla_gqa_dims *dims, int32_t batch, int32_t q_len, int32_t max_kv_len,
                                  int32_t num_splits, size_t *o_part_bytes, size_t *lse_part_bytes,
                                  int32_t *num_splits_used);

/* One decode step of GQA attention, split over the units' 128-token tiles and
 * merged: for query i of sequence b at p = kv_len[b] - q_len + i and head h
 * of group g = h / (H/G),
 *   o = sum_j softmax_j(sm_scale (R_p q[b,i,h]) . K[b,g,j]) V[b,g,j],  j <= p
 * q [batch, q_len, H, head_dim] bf16 (not rotated), q_len * H/G <= 128;
 * o_part / lse_part sized by mla_gqa_workspace_size; outputs
 * o [batch, q_len, H, head_dim] fp32, lse [batch, q_len, H] fp32 (natural
 * log) or NULL. */
mla_status mla_gqa_decode_attn(const mla_gqa_dims *dims, const mla_cache *cache, int32_t batch, int32_t q_len,
                               const int32_t *kv_len, int32_t max_kv_len, const void *q, int32_t num_splits,
                               float *o_part, float *lse_part, float *o, float *lse, void *stream);

/* Projections of the original GQA layer (Sec. 3.1, Eq. 1), bf16 results:
 *   q [batch, n_new, H, head_dim]         = h W_Q^T   (W_Q [H head_dim, hidden])
 *   k_new, v_new [batch, n_new, G, head_dim] = h W_K^T, h W_V^T (W_K, W_V [G head_dim, hidden])
 * h [batch, n_new, hidden] bf16, hidden a multiple of 8; every pointer 16-byte
 * aligned.  (q is not rotated; mla_gqa_append rotates the keys, the attention
 * the queries.) */
mla_status mla_gqa_project(const mla_gqa_dims *dims, int32_t batch, int32_t n_new, int32_t hidden, const void *h,
                           const void *w_q, const void *w_k, const void *w_v, void *q, void *k_new, void *v_new,
                           void *stream);

/* Output projection of the original GQA layer: out [batch, q_len, hidden] =
 * W_O concat_h o (concat index h head_dim + e), o [batch, q_len, H, head_dim]
 * fp32 (as mla_gqa_decode_attn writes it), W_O [hidden, H head_dim] bf16; the
 * same frozen W_O serves the converted MLA layer (Sec. 4.1). */
mla_status mla_gqa_out_proj(const mla_gqa_dims *dims, int32_t batch, int32_t q_len, int32_t hidden, const float *o,
                            const void *w_o, void *out, void *stream);

/* Forward value of the E2E functional-reconstruction loss of one layer
 * (Sec. 4.1): the masked mean-squared error between the converted MLA
 * block's post-W_O output and the frozen original block's,
 *   loss = sum_t M_t sum_d (a_mla[t, d] - a_orig[t, d])^2 / (hidden sum_t M_t)
 * a_mla, a_orig [rows, hidden] bf16 (hidden a multiple of 8, 16-byte
 * aligned); mask [rows] uint8 (nonzero = counted) or NULL (every row); loss:
 * one device float (0 when no row counts).  fp32 products, fp64 sums, added
 * in a fixed order: the same bits on every run.  Backward and training are
 * not part of this library. */
mla_status mla_e2e_loss(int32_t rows, int32_t hidden, const void *a_mla, const void *a_orig, const uint8_t *mask,
                        float *loss, void *stream);

/* mla_decode_attn followed by mla_combine, for callers that cannot allocate
 * device memory: code that runs where an allocation is not allowed (inside a
 * runtime that owns all device memory through its own pool, in an inference
 * path whose memory budget is fixed up front, or in a plugin handed only its
 * input and output tensors).  It allocates nothing and takes no partial
 * buffers: the split partials go to one array of 32 MiB that the library
 * reserves statically on every device that loads it, for the life of the
 * process.  The paper has no counterpart; this is a property of the library.
 *   Inputs as for mla_decode_attn; outputs o_lat [batch, q_len, H, rank] fp32
 *   and lse [batch, q_len, H] fp32 (or NULL), as mla_combine writes them.
 *   num_splits > 0 is used as given; 0 picks the usual automatic count,
 *   lowered if needed so that (batch + S - 1) * q_len * H * (rank + 1) floats
 *   fit the array.  A size that cannot fit returns MLA_ERR_UNSUPPORTED
 *   before anything is launched.
 *   The first call on a device looks up the array's device address with that
 *   device current (a host-side query); make that first call before any stream
 *   capture.  Every call uses the same array, so calls that overlap on the GPU
 *   (different streams, or different threads) race and must be serialised.
 *   Nothing in the array has to start at zero: each call writes the partial
 *   of every (sequence, partition) pair that holds tiles before its combine
 *   reads it.  The slots of empty partitions (fewer tiles than partitions)
 *   may hold stale data from an earlier call; the combine loads them but
 *   gives them zero weight, so they never reach an output. */
mla_status mla_decode_attn_noalloc(const mla_dims *dims, const mla_cache *cache, int32_t batch, int32_t q_len,
                                   const int32_t *kv_len, int32_t max_kv_len, const void *q_abs, int32_t num_splits,
                                   float *o_lat, float *lse, void *stream);

/* Synchronise `stream`, then read and clear the current device's sticky
 * status word: MLA_OK, MLA_ERR_DEVICE_BOUNDS or MLA_ERR_DEVICE_TIMEOUT
 * (MLA_ERR_CUDA if the synchronisation itself failed). */
mla_status mla_check_status(void *stream);

/* Self-test of the bounded-wait machinery: launches one block that waits on
 * an mbarrier nothing ever signals, with a limit of `limit_ns` nanoseconds
 * (clamped to [1e3, 1e9]); the wait must run out and record
 * MLA_ERR_DEVICE_TIMEOUT.  Returns the launch status only; read the outcome
 * with mla_check_status(). */
mla_status mla_selftest_wait_timeout(int64_t limit_ns, void *stream);

/* Testing aid: re-read the GBMLA_* environment variables that choose the
 * kernels' tiling (they are otherwise read once per process, at the first
 * call that needs them): GBMLA_ATTN_KERNEL=simt (CUDA-core attention),
 * GBMLA_TC_MAX_N (query rows per tensor-core CTA, 16..80), GBMLA_TC_MAX_SLOTS
 * and GBMLA_TC_PV_SLOTS (ring slots), GBMLA_TC_QUERY=resident|streamed (an
 * 80-row tensor-core CTA keeps its queries in shared memory or loads them with
 * each cache chunk), GBMLA_ABSORB=persistent|gemm (the absorption kernel, where
 * both serve the shape).  Results are the same under
 * every setting, up to the floating-point order of the split partials.  Not
 * thread-safe against concurrent launches; the paper has no counterpart. */
void mla_reload_tuning(void);

/* Text of the CUDA error behind the last MLA_ERR_CUDA returned to the calling
 * thread ("" if none).  The library's own; it has no counterpart in the
 * paper. */
const char *mla_last_error(void);

/* Static name of a status code. */
const char *mla_status_str(mla_status status);

#ifdef __cplusplus
}
#endif
#endif /* GBMLA_H */
