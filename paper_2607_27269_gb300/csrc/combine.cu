// mla_combine: merge the split-KV partials of each sequence with their
// log-sum-exp weights (the softmax normaliser of Eq. 3).
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace gbmla {
namespace {

// Block (row group, sequence b), 128 threads.  A row of o_lat is rank floats;
// each thread owns one float4 of it (rank / 4 threads per row) in RPT rows
// (RPT > 1 only when there are rows enough to fill the GPU anyway: it spreads
// the per-block prologue over more work).  The partials are merged online:
// KF partitions per step, their log-sum-exps and partial rows all loaded
// together, the running exponent base raised when a step brings a larger one.
// An empty partition (fewer tiles than partitions) was never written: its
// values are loaded (the slot exists) but never used.
constexpr int kCombineThreads = 128;

template <int RPT, int KF>
__global__ void __launch_bounds__(kCombineThreads) combine_kernel(int batch, int q_len, int H, int rank, int max_kv,
                                                                 int S, const int32_t *__restrict__ kv_len,
                                                                 const float *__restrict__ o_part,
                                                                 const float *__restrict__ lse_part, float *o_lat,
                                                                 float *lse_out, int groups)
{
    griddep_wait();
    griddep_launch_dependents();
    __shared__ int64_t red[64];
    const int b = blockIdx.y;  // unit b: sequence b / groups (groups > 1: one unit per KV group)
    int64_t T, t0;
    block_tile_sums(kv_len, batch, b, q_len, max_kv, red, &T, &t0, groups);
    const int64_t nb = seq_tiles(kv_len[b / groups], q_len, max_kv);
    if (nb == 0 || T == 0) return;  // invalid length: recorded by the attention kernel
    const int k_first = part_of_tile(t0, T, S), k_last = part_of_tile(t0 + nb - 1, T, S);
    const int rows = q_len * H;
    const int tpr = rank / 4, rpb = kCombineThreads / tpr;
    const int part = threadIdx.x % tpr;
    if (threadIdx.x >= rpb * tpr) return;  // rank / 4 need not divide the block
    const int row0 = blockIdx.x * rpb * RPT + threadIdx.x / tpr;
    const bool may_be_empty = T < S;  // a partition is empty only when there are fewer tiles than partitions
    float m[RPT], wsum[RPT];
    float4 acc[RPT];
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
        m[r] = -INFINITY;
        wsum[r] = 0.f;
        acc[r] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    for (int k0 = k_first; k0 <= k_last; k0 += KF) {
        float l[RPT][KF];
        float4 x[RPT][KF];
#pragma unroll
        for (int j = 0; j < KF; ++j) {
            const int k = k0 + j;
            const bool live = k <= k_last && !(may_be_empty && part_begin(k, T, S) == part_begin(k + 1, T, S));
            const int64_t slot = static_cast<int64_t>(b) + (k <= k_last ? k : k_last);
#pragma unroll
            for (int r = 0; r < RPT; ++r) {
                const int row = row0 + r * rpb;
                l[r][j] = -INFINITY;
                x[r][j] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (row < rows) {
                    const float lv = lse_part[slot * rows + row];
                    x[r][j] = __ldcs(reinterpret_cast<const float4 *>(o_part + (slot * rows + row) * rank) + part);
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
            acc[r].x *= sc;
            acc[r].y *= sc;
            acc[r].z *= sc;
            acc[r].w *= sc;
#pragma unroll
            for (int j = 0; j < KF; ++j) {
                if (l[r][j] == -INFINITY) continue;  // no key there, or never written
                const float wk = __expf(l[r][j] - mn);
                wsum[r] += wk;
                acc[r].x += wk * x[r][j].x;
                acc[r].y += wk * x[r][j].y;
                acc[r].z += wk * x[r][j].z;
                acc[r].w += wk * x[r][j].w;
            }
        }
    }
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
        const int row = row0 + r * rpb;
        if (row >= rows) continue;
        const float inv = wsum[r] > 0.f ? 1.f / wsum[r] : 0.f;
        // output row: (b, row) for the MLA path; for groups > 1, row = i * H + head of
        // sequence b / groups, head = (b % groups) * H + h (rows of a unit are (i, h))
        const int64_t orow = groups == 1 ? static_cast<int64_t>(b) * rows + row
                                         : (static_cast<int64_t>(b / groups) * q_len + row / H) * (groups * H) +
                                               (b % groups) * H + row % H;
        reinterpret_cast<float4 *>(o_lat + orow * rank)[part] =
            make_float4(acc[r].x * inv, acc[r].y * inv, acc[r].z * inv, acc[r].w * inv);
        if (lse_out && part == 0) lse_out[orow] = wsum[r] > 0.f ? m[r] + logf(wsum[r]) : -INFINITY;
    }
}

}  // namespace

cudaError_t launch_combine(int batch, int q_len, int num_heads, int rank, int max_kv, int num_splits,
                           const int32_t *kv_len, const float *o_part, const float *lse_part, float *o_lat,
                           float *lse, cudaStream_t st, int groups)
{
    // rank is a multiple of 64 (<= 512): rank / 4 <= 128 threads per row
    const int tpr = rank / 4, rpb = kCombineThreads / tpr;
    const int rows = q_len * num_heads;
    if (batch == 0 || rows == 0) return cudaSuccess;
    // four rows per thread once that still leaves several blocks per SM
    const int64_t blocks1 = static_cast<int64_t>((rows + rpb - 1) / rpb) * batch;
    if (blocks1 >= 16 * 152) {
        dim3 grid((rows + 4 * rpb - 1) / (4 * rpb), batch);
        return launch_dependent(combine_kernel<4, 2>, grid, dim3(kCombineThreads), 0, st, 1, batch, q_len, num_heads,
                                rank, max_kv, num_splits, kv_len, o_part, lse_part, o_lat, lse, groups);
    }
    dim3 grid((rows + rpb - 1) / rpb, batch);
    return launch_dependent(combine_kernel<1, 8>, grid, dim3(kCombineThreads), 0, st, 1, batch, q_len, num_heads, rank,
                            max_kv, num_splits, kv_len, o_part, lse_part, o_lat, lse, groups);
}

}  // namespace gbmla
