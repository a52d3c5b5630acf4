// CUDA-core split-KV attention core over the latent cache (Eqs. 2-4 with the
// Sec. 3.3 score routing, in the absorbed form).  A plain, generic kernel:
// every (partition, group of kSimtRows query rows) block re-reads its cache
// tiles, scores them with fp32 FMAs and keeps an online softmax.
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace gbmla {
namespace {

constexpr int kRows = kSimtRows;  // query rows per block
constexpr int kTok = 32;          // tokens per inner tile
constexpr int kThreads = 256;
constexpr int kMaxCols = 2;       // rank <= 512 = kThreads * kMaxCols

struct Smem {
    int64_t red[32];
    float m[kRows], l[kRows], alpha[kRows];
    float s[kRows][kTok];
    int tok_ok[kTok];
};

__global__ void __launch_bounds__(kThreads) attn_simt_kernel(AttnArgs a)
{
    griddep_wait();
    griddep_launch_dependents();
    extern __shared__ __align__(16) unsigned char dyn[];
    __shared__ Smem sm;
    const int K = a.rank + a.d_rope;
    const int KP = K + 2;  // padded bf16 row stride of the key tile (bank spread)
    const int QP = K + 1;  // padded fp32 row stride of the query tile
    float *qs = reinterpret_cast<float *>(dyn);                                       // [kRows][QP]
    uint16_t *ks = reinterpret_cast<uint16_t *>(dyn + sizeof(float) * kRows * QP);    // [kTok][KP]

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int rows = a.q_len * a.num_heads;
    const int row0 = blockIdx.y * kRows;
    const int nrows = min(kRows, rows - row0);
    const int part = blockIdx.x;
    const CacheView &c = a.cache;
    const float scale_log2 = a.sm_scale * 1.4426950408889634f;

    if (part == 0 && blockIdx.y == 0) {
        // unusable lengths hold no tiles anywhere; record them once
        for (int bb = tid; bb < a.batch; bb += kThreads) {
            const int kv = a.kv_len[bb];
            if (kv < a.q_len || kv > a.max_kv) record_status(a.status, kStatusBounds);
        }
    }
    const int64_t T = block_tile_sum(a.kv_len, a.batch, a.q_len, a.max_kv, sm.red);
    if (T == 0) return;
    const int64_t t_begin = part_begin(part, T, a.num_splits), t_end = part_begin(part + 1, T, a.num_splits);
    if (t_begin >= t_end) return;

    int64_t cum = 0;
    for (int b = 0; b < a.batch && cum < t_end; ++b) {
        const int kv = a.kv_len[b];
        const int64_t nb = seq_tiles(kv, a.q_len, a.max_kv);
        const int64_t s0 = max(cum, t_begin), s1 = min(cum + nb, t_end);
        cum += nb;
        if (s0 >= s1) continue;
        // ---- this sequence's segment: tokens [tok_lo, tok_hi)
        const int tok_lo = static_cast<int>((s0 - (cum - nb)) * MLA_SPLIT_TILE);
        const int tok_hi = min(kv, static_cast<int>((s1 - (cum - nb)) * MLA_SPLIT_TILE));
        const uint16_t *qsrc = static_cast<const uint16_t *>(a.q_abs) + (static_cast<int64_t>(b) * rows + row0) * K;
        for (int e = tid; e < kRows * K; e += kThreads) {
            const int r = e / K;
            qs[r * QP + e % K] = r < nrows ? bf16_bits_to_float(qsrc[e]) : 0.f;
        }
        if (tid < kRows) {
            sm.m[tid] = -INFINITY;
            sm.l[tid] = 0.f;
        }
        float acc[kRows][kMaxCols];
#pragma unroll
        for (int r = 0; r < kRows; ++r)
#pragma unroll
            for (int u = 0; u < kMaxCols; ++u) acc[r][u] = 0.f;
        __syncthreads();

        for (int t0 = tok_lo; t0 < tok_hi; t0 += kTok) {
            // ---- load the key tile [c_j | k_rope_j] for kTok tokens
            for (int e = tid; e < kTok * (K / 8); e += kThreads) {
                const int j = e / (K / 8), v = e % (K / 8);
                const int64_t t = t0 + j;
                uint4 val = make_uint4(0, 0, 0, 0);
                bool ok = t < tok_hi;
                if (ok) {
                    int64_t blk = b, slot = t;
                    if (c.block_table) {
                        const int32_t page = c.block_table[static_cast<int64_t>(b) * c.bt_stride + t / c.page_size];
                        if (page < 0 || page >= c.num_pages) {
                            ok = false;
                            record_status(a.status, kStatusBounds);
                        }
                        blk = page;
                        slot = t % c.page_size;
                    }
                    if (ok) {
                        const int col = v * 8;
                        const uint16_t *src = col < a.rank
                                                  ? (const uint16_t *)c.c_kv + blk * c.c_blk + slot * c.c_tok + col
                                                  : (const uint16_t *)c.k_rope + blk * c.r_blk + slot * c.r_tok +
                                                        (col - a.rank);
                        val = *reinterpret_cast<const uint4 *>(src);
                    }
                }
                uint32_t *dst = reinterpret_cast<uint32_t *>(ks + j * KP + v * 8);
                dst[0] = val.x;
                dst[1] = val.y;
                dst[2] = val.z;
                dst[3] = val.w;
                if (v == 0) sm.tok_ok[j] = ok;
            }
            __syncthreads();
            // ---- scores: thread -> (row, two tokens)
            {
                const int r = tid / 16, j0 = tid % 16;
#pragma unroll
                for (int jj = 0; jj < 2; ++jj) {
                    const int j = j0 + 16 * jj;
                    const float *q = qs + r * QP;
                    const uint32_t *k2 = reinterpret_cast<const uint32_t *>(ks + j * KP);
                    float dot = 0.f;
                    for (int e = 0; e < K / 2; ++e) {
                        const uint32_t w = k2[e];
                        dot = fmaf(q[2 * e], __uint_as_float(w << 16), dot);
                        dot = fmaf(q[2 * e + 1], __uint_as_float(w & 0xffff0000u), dot);
                    }
                    const int i = (row0 + r) / a.num_heads;
                    const int pos = t0 + j;
                    const bool vis = r < nrows && sm.tok_ok[j] && pos <= kv - a.q_len + i;
                    sm.s[r][j] = vis ? dot * scale_log2 : -INFINITY;
                }
            }
            __syncthreads();
            // ---- online softmax (log2 domain), one warp per two rows
            for (int r = warp; r < kRows; r += kThreads / 32) {
                const float s = sm.s[r][lane];
                float tmax = s;
                for (int o = 16; o > 0; o >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
                const float m_old = sm.m[r];
                const float m_new = fmaxf(m_old, tmax);
                const float base = m_new == -INFINITY ? 0.f : m_new;
                const float p = s == -INFINITY ? 0.f : exp2f(s - base);
                float psum = p;
                for (int o = 16; o > 0; o >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, o);
                sm.s[r][lane] = p;
                __syncwarp();
                if (lane == 0) {
                    const float al = m_old == -INFINITY ? 0.f : exp2f(m_old - base);
                    sm.alpha[r] = al;
                    sm.l[r] = sm.l[r] * al + psum;
                    sm.m[r] = m_new;
                }
            }
            __syncthreads();
            // ---- O = alpha * O + P . C
#pragma unroll
            for (int u = 0; u < kMaxCols; ++u) {
                const int col = tid + u * kThreads;
                if (col < a.rank) {
                    float cv[kTok];
#pragma unroll
                    for (int j = 0; j < kTok; ++j) cv[j] = bf16_bits_to_float(ks[j * KP + col]);
#pragma unroll
                    for (int r = 0; r < kRows; ++r) {
                        float v = acc[r][u] * sm.alpha[r];
#pragma unroll
                        for (int j = 0; j < kTok; ++j) v = fmaf(sm.s[r][j], cv[j], v);
                        acc[r][u] = v;
                    }
                }
            }
            __syncthreads();
        }
        // ---- write this sequence's partial
        const int64_t slot = static_cast<int64_t>(b) + part;
#pragma unroll
        for (int u = 0; u < kMaxCols; ++u) {
            const int col = tid + u * kThreads;
            if (col < a.rank) {
#pragma unroll
                for (int r = 0; r < kRows; ++r) {
                    if (r < nrows) {
                        const float l = sm.l[r];
                        a.o_part[(slot * rows + row0 + r) * a.rank + col] = l > 0.f ? acc[r][u] / l : 0.f;
                    }
                }
            }
        }
        if (tid < nrows) {
            const float l = sm.l[tid];
            a.lse_part[slot * rows + row0 + tid] = l > 0.f ? (sm.m[tid] + log2f(l)) * 0.69314718055994531f : -INFINITY;
        }
        __syncthreads();
    }
}

}  // namespace

cudaError_t launch_attn_simt(const AttnArgs &a, cudaStream_t st)
{
    const int K = a.rank + a.d_rope;
    const size_t smem = sizeof(float) * kRows * (K + 1) + sizeof(uint16_t) * kTok * (K + 2);
    cudaError_t e = cudaFuncSetAttribute(attn_simt_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    const int rows = a.q_len * a.num_heads;
    dim3 grid(a.num_splits, (rows + kRows - 1) / kRows);
    cudaError_t e0 = launch_dependent(attn_simt_kernel, grid, dim3(kThreads), smem, st, 1, a);
    if (e0 != cudaSuccess) return e0;
    return cudaGetLastError();
}

}  // namespace gbmla
