// mla_combine: merge the split-KV partials of each sequence with their
// log-sum-exp weights (the softmax normaliser of Eq. 3).
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace gbmla {
namespace {

// Block (row block, unit b), 256 threads.  A row of o_lat is rank floats;
// each thread owns eight consecutive floats of it (two float4; rank / 8
// threads per row).  The threads form SG slot groups of 256 / SG threads;
// a group holds rows side by side, RPT rows per thread.  Each group merges its
// share of the unit's partitions (k_first + sg, + SG, ...) online: KF of them
// per step, their log-sum-exps and partial rows all loaded together, the
// running exponent base raised when a step brings a larger one.  With SG > 1
// (many partitions per sequence: few sequences over many SMs) the groups'
// merge states then meet in shared memory and group 0 finishes; the per-warp
// chain of dependent loads and exponentials is what bounds this kernel, so
// splitting the partitions over more warps shortens it.  An empty partition
// (fewer tiles than partitions) was never written: its values are never used.
constexpr int kCombineThreads = 256;

template <int RPT, int KF, int SG>
__global__ void __launch_bounds__(kCombineThreads) combine_kernel(int batch, int q_len, int H, int rank, int max_kv,
                                                                 int S, const int32_t *__restrict__ kv_len,
                                                                 const float *__restrict__ o_part,
                                                                 const float *__restrict__ lse_part, float *o_lat,
                                                                 float *lse_out, int groups, int skip_whole)
{
    static_assert(SG == 1 || RPT == 1, "slot groups merge one row per thread");
    griddep_wait();
    griddep_launch_dependents();
    __shared__ int64_t red[64];
    __shared__ float xs[SG > 1 ? kCombineThreads * 10 : 1];
    const int b = blockIdx.y;  // unit b: sequence b / groups (groups > 1: one unit per KV group)
    int64_t T, t0;
    block_tile_sums(kv_len, batch, b, q_len, max_kv, red, &T, &t0, groups);
    const int64_t nb = seq_tiles(kv_len[b / groups], q_len, max_kv);
    if (nb == 0 || T == 0) return;  // invalid length: recorded by the attention kernel
    const int k_first = part_of_tile(t0, T, S), k_last = part_of_tile(t0 + nb - 1, T, S);
    if (skip_whole && k_first == k_last) return;  // its one partition wrote the final rows itself
    const int rows = q_len * H;
    const int tpr = rank / 8, gsz = kCombineThreads / SG, rpg = gsz / tpr;
    const int sg = threadIdx.x / gsz, t = threadIdx.x % gsz;
    const int part = t % tpr, rr = t / tpr;
    const bool active = rr < rpg;  // (tpr need not divide the group)
    const bool may_be_empty = T < S;  // a partition is empty only when there are fewer tiles than partitions
    // Row blocks blockIdx.x, + gridDim.x, ... of the unit (one per block with
    // slot groups, whose finishing group alone goes on past the merge).
    const int nrb = (rows + rpg * RPT - 1) / (rpg * RPT);
    for (int rb = blockIdx.x; rb < nrb; rb += gridDim.x) {
    const int row0 = rb * rpg * RPT + rr;
    float m[RPT], wsum[RPT], acc[RPT][8];
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
        m[r] = -INFINITY;
        wsum[r] = 0.f;
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[r][e] = 0.f;
    }
    if (active) {
        for (int k0 = k_first + sg; k0 <= k_last; k0 += SG * KF) {
            float l[RPT][KF];
            float4 x[RPT][KF][2];
#pragma unroll
            for (int j = 0; j < KF; ++j) {
                const int k = k0 + j * SG;
                const bool in = k <= k_last;
                const bool live = in && !(may_be_empty && part_begin(k, T, S) == part_begin(k + 1, T, S));
                const int64_t slot = static_cast<int64_t>(b) + (in ? k : k_last);
#pragma unroll
                for (int r = 0; r < RPT; ++r) {
                    const int row = row0 + r * rpg;
                    l[r][j] = -INFINITY;
                    x[r][j][0] = x[r][j][1] = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (in && row < rows) {
                        const float lv = lse_part[slot * rows + row];
                        const float4 *src = reinterpret_cast<const float4 *>(o_part + (slot * rows + row) * rank) + 2 * part;
                        x[r][j][0] = __ldcs(src);
                        x[r][j][1] = __ldcs(src + 1);
                        l[r][j] = live ? lv : -INFINITY;
                    }
                }
            }
#pragma unroll
            for (int r = 0; r < RPT; ++r) {
                float bm = l[r][0];
#pragma unroll
                for (int j = 1; j < KF; ++j) bm = fmaxf(bm, l[r][j]);
                if (bm == -INFINITY) continue;
                const float mn = fmaxf(m[r], bm);
                const float sc = m[r] == -INFINITY ? 0.f : __expf(m[r] - mn);
                m[r] = mn;
                wsum[r] *= sc;
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[r][e] *= sc;
#pragma unroll
                for (int j = 0; j < KF; ++j) {
                    if (l[r][j] == -INFINITY) continue;  // no key there, or never written
                    const float wk = __expf(l[r][j] - mn);
                    wsum[r] += wk;
                    const float xv[8] = {x[r][j][0].x, x[r][j][0].y, x[r][j][0].z, x[r][j][0].w,
                                         x[r][j][1].x, x[r][j][1].y, x[r][j][1].z, x[r][j][1].w};
#pragma unroll
                    for (int e = 0; e < 8; ++e) acc[r][e] += wk * xv[e];
                }
            }
        }
    }
    if constexpr (SG > 1) {
        float *st = xs + threadIdx.x * 10;
        st[0] = m[0];
        st[1] = wsum[0];
#pragma unroll
        for (int e = 0; e < 8; ++e) st[2 + e] = acc[0][e];
        __syncthreads();
        if (sg != 0) return;
        float mx = m[0];
#pragma unroll
        for (int g = 1; g < SG; ++g) mx = fmaxf(mx, xs[(g * gsz + t) * 10]);
        if (mx != -INFINITY) {
            const float s0 = __expf(m[0] - mx);  // 0 for a group that merged nothing
            wsum[0] *= s0;
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[0][e] *= s0;
#pragma unroll
            for (int g = 1; g < SG; ++g) {
                const float *o = xs + (g * gsz + t) * 10;
                const float sc = __expf(o[0] - mx);
                wsum[0] += sc * o[1];
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[0][e] += sc * o[2 + e];
            }
        }
        m[0] = mx;
    }
    if (!active) continue;
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
        const int row = row0 + r * rpg;
        if (row >= rows) continue;
        const float inv = wsum[r] > 0.f ? 1.f / wsum[r] : 0.f;
        // output row: (b, row) for the MLA path; for groups > 1, row = i * H + head of
        // sequence b / groups, head = (b % groups) * H + h (rows of a unit are (i, h))
        const int64_t orow = groups == 1 ? static_cast<int64_t>(b) * rows + row
                                         : (static_cast<int64_t>(b / groups) * q_len + row / H) * (groups * H) +
                                               (b % groups) * H + row % H;
        float4 *dst = reinterpret_cast<float4 *>(o_lat + orow * rank) + 2 * part;
        dst[0] = make_float4(acc[r][0] * inv, acc[r][1] * inv, acc[r][2] * inv, acc[r][3] * inv);
        dst[1] = make_float4(acc[r][4] * inv, acc[r][5] * inv, acc[r][6] * inv, acc[r][7] * inv);
        if (lse_out && part == 0) lse_out[orow] = wsum[r] > 0.f ? m[r] + logf(wsum[r]) : -INFINITY;
    }
    }
}

}  // namespace

cudaError_t launch_combine(int batch, int q_len, int num_heads, int rank, int max_kv, int num_splits,
                           const int32_t *kv_len, const float *o_part, const float *lse_part, float *o_lat,
                           float *lse, cudaStream_t st, int groups, bool skip_whole)
{
    // rank is a multiple of 64 (<= 512): rank / 8 <= 64 threads per row
    const int tpr = rank / 8;
    const int rows = q_len * num_heads;
    if (batch == 0 || rows == 0) return cudaSuccess;
    // Blocks per unit.  With one row block each, the partition prologue (a
    // reduction over every sequence's tile count) is repeated per row block;
    // so a block of a single-group kernel takes up to four row blocks, as
    // many as still leave four blocks per SM.  (Measured on the 128-sequence
    // paged batch: the step 362.7 -> 358.7 us with four; with four row
    // blocks on the 32-sequence chunk batch the combine went 9.4 -> 12.2 us.)
    auto go = [&](auto kernel, int rows_per_block, bool looped) {
        const int nrb = (rows + rows_per_block - 1) / rows_per_block;
        int per = 1;
        if (looped)
            while (per < 4 && static_cast<int64_t>(nrb) * batch >= static_cast<int64_t>(per + 1) * 4 * 152) ++per;
        dim3 grid((nrb + per - 1) / per, batch);
        return launch_dependent(kernel, grid, dim3(kCombineThreads), 0, st, 1, batch, q_len, num_heads, rank, max_kv,
                                num_splits, kv_len, o_part, lse_part, o_lat, lse, groups, skip_whole ? 1 : 0);
    };
    // Many partitions per unit (a few long sequences spread over the SMs):
    // slot groups of the smallest whole number of warps that holds a row.
    if (num_splits >= 4 * batch) {
        const int gsz = (tpr + 31) / 32 * 32;
        if (kCombineThreads / gsz >= 8) return go(combine_kernel<1, 4, 8>, (kCombineThreads / 8) / tpr, false);
        return go(combine_kernel<1, 4, 4>, (kCombineThreads / 4) / tpr, false);
    }
    // Few partitions per unit: rows side by side, two rows per thread once
    // that still leaves several blocks per SM
    const int rpb = kCombineThreads / tpr;
    if (static_cast<int64_t>((rows + rpb - 1) / rpb) * batch >= 8 * 152) return go(combine_kernel<2, 2, 1>, 2 * rpb, true);
    return go(combine_kernel<1, 4, 1>, rpb, true);
}

}  // namespace gbmla
