// Host-side declarations shared by the C-ABI glue (api.cu) and the kernel
// translation units.  Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/gbmla.h"

namespace gbmla {

// Cache description as the kernels take it (validated by api.cu).
struct CacheView {
    const void *c_kv;
    const void *k_rope;
    int64_t c_tok, r_tok, c_blk, r_blk;   // strides in elements
    const int32_t *block_table;           // nullptr: contiguous
    int32_t bt_stride, page_size, num_pages, capacity;
};

struct AttnArgs {
    int32_t batch, q_len, num_heads, rank, d_rope;
    float sm_scale;
    const int32_t *kv_len;
    int32_t max_kv;         // lengths above this (<= capacity) are unusable
    const void *q_abs;      // bf16 [B, q, H, rank + d_rope]
    int32_t num_splits;     // S (resolved)
    float *o_part, *lse_part;
    // tensor-core kernel only, or NULL: a sequence whose tiles all lie in one
    // partition writes its final output / log-sum-exp rows here ([B, q, H, rank]
    // and [B, q, H], as mla_combine writes them) instead of its partial slot;
    // the combine then skips it (launch_combine's skip_whole)
    float *o_final = nullptr, *lse_final = nullptr;
    CacheView cache;
    unsigned *status;
};

// groups > 1: `batch` counts (sequence, KV group) units, entry rows
// [sequence, n_new, group, .] (token-major, as a projection writes them),
// start_pos indexed by sequence (unit / groups); rank = value width, d_rope =
// key width (the original-GQA cache).
cudaError_t launch_append(const mla_dims &d, const CacheView &c, int batch, int n_new, const void *c_new,
                          const void *kr_new, const int32_t *start_pos, unsigned *status, cudaStream_t st,
                          int groups = 1);

cudaError_t launch_absorb(const mla_dims &d, int batch, int q_len, const void *q_nope, const void *q_pe,
                          const int32_t *kv_len, const void *w_uk, void *q_abs, unsigned *status,
                          cudaStream_t st);

// CUDA-core attention core; `qgroups` query groups of kSimtRows rows each.
constexpr int kSimtRows = 16;
cudaError_t launch_attn_simt(const AttnArgs &a, cudaStream_t st);

// Testing aids, read from the environment once per process (and again by
// mla_reload_tuning): GBMLA_ATTN_KERNEL=simt (attn_simt = 1) forces the
// CUDA-core attention; GBMLA_TC_MAX_N caps the query rows per tensor-core CTA;
// GBMLA_TC_MAX_SLOTS caps its ring slots and GBMLA_TC_PV_SLOTS sets the share
// of the value-product ring; GBMLA_ABSORB=persistent|gemm (absorb_path 1|2)
// chooses the absorption kernel where both serve the shape;
// GBMLA_TC_QUERY=resident|streamed (tc_query 1|2) keeps the queries of an
// 80-row tensor-core CTA in shared memory or streams them with the cache
// chunks.  0 means "not set".  They change tiling only.
struct Tuning {
    int attn_simt, tc_max_rows, tc_max_slots, tc_pv_slots, absorb_path, tc_query;
};
const Tuning &tuning();
void reload_tuning();

// Tensor-core attention core (tcgen05 + TMA).  For q_len * num_heads query
// rows it runs `groups` independent CTAs of `n` rows per partition.
struct TcShape {
    int n, groups;
};
TcShape attn_tc_shape(int rows);
cudaError_t launch_attn_tc(const AttnArgs &a, cudaStream_t st);

// `groups` > 1: unit b of `batch` is KV group b % groups of sequence b / groups
// (the original-GQA path; num_heads = heads per group); its length is
// kv_len[b / groups], and its rows (i, h) go to head (b % groups) * num_heads + h
// of row (sequence, i) of o_lat / lse, i.e. [B, q_len, G * num_heads, rank].
cudaError_t launch_combine(int batch, int q_len, int num_heads, int rank, int max_kv, int num_splits,
                           const int32_t *kv_len, const float *o_part, const float *lse_part, float *o_lat,
                           float *lse, cudaStream_t st, int groups = 1, bool skip_whole = false);

cudaError_t launch_out_proj(const mla_dims &d, int batch, int q_len, const float *o_lat, const void *w_uv,
                            const void *w_o, void *o, void *out, unsigned *status, cudaStream_t st);

// Grouped GEMM of the projections: for each group g < G and row m < M,
// C[phys(g, m), n] = sum_k A[phys(g, m), k] B_g(n, k) (bf16 result), with
// phys(g, m) = (m / hpg) * blk + g * hpg + m % hpg.  A is fp32 or bf16 with
// row stride lda; B_g(n, k) = B[g N K + n K + k] (K-major) or B[g K N + k N + n]
// (N-major), bf16.  K and N are multiples of 8; A, B and C 16-byte aligned;
// hpg <= 128 divides M.
struct GroupGemm {
    int M, N, K, G;
    int hpg, blk;
    const void *A;
    int a_f32;
    int64_t lda;
    const void *B;
    int b_nmajor;
    void *C;
    int64_t ldc;
    unsigned *status;
    int stages, rblk, ksplit;  // set by the launcher
    int a_stride;              // bytes between A ring stages (set by the launcher)
};
cudaError_t launch_group_gemm(const GroupGemm &p, cudaStream_t st);
// The absorption GEMM (N-major W_UK, bf16 A) that also writes the rotated
// positional query into columns [rank, rank + d_rope) of its output rows.
cudaError_t launch_absorb_gemm(const GroupGemm &p, const mla_dims &d, const void *q_pe, const int32_t *kv_len,
                               int q_len, cudaStream_t st);

// Projection of the step's hidden states (mla_project_append): one GEMM of
// h [batch * n_new, hidden] with the three weights side by side, whose
// epilogue writes the latent rows and the rotated positional keys into the
// cache and the two query parts to q_nope / q_pe.
cudaError_t launch_project(const mla_dims &d, const CacheView &c, int batch, int n_new, const void *h,
                           const void *w_dkv, const void *w_kr, const void *w_q, const int32_t *start_pos,
                           void *q_nope, void *q_pe, unsigned *status, cudaStream_t st);

// Acceptance statistics (mla_acceptance_stats): dtype 0 = fp32, 1 = bf16 logits.
cudaError_t launch_acceptance(int rows, int vocab, int dtype, const void *draft, const void *target, int64_t stride,
                              float *alpha, int32_t *argmax_d, int32_t *argmax_t, int32_t *greedy, unsigned *status,
                              cudaStream_t st);

// Original-GQA decode attention (mla_gqa_decode_attn): per (sequence, KV
// group) unit b * G + g, keys in cache.k_rope and values in cache.c_kv.
struct GqaLaunch {
    int batch, q_len, groups, hpg, head_dim, max_kv, num_splits;
    float sm_scale;
    int rope_style;
    float rope_base;
    const int32_t *kv_len;
    const void *q;        // bf16 [B, q_len, H, head_dim], not rotated
    float *o_part, *lse_part;
    unsigned *status;
    CacheView cache;
};
cudaError_t launch_gqa_attn(const GqaLaunch &g, cudaStream_t st);

// E2E loss forward (mla_e2e_loss): a_mla, a_orig bf16 [rows, hidden], mask [rows] or null.
cudaError_t launch_e2e_loss(int rows, int hidden, const void *a_mla, const void *a_orig, const uint8_t *mask,
                            float *loss, cudaStream_t st);

cudaError_t launch_selftest_wait(int64_t limit_ns, unsigned *status, cudaStream_t st);

}  // namespace gbmla
