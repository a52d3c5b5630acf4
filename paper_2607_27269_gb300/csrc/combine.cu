// mla_combine: merge the split-KV partials of each sequence with their
// log-sum-exp weights (the softmax normaliser of Eq. 3).
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace gbmla {
namespace {

// One block per sequence, one warp per (i, h) row.  Every lane owns up to 4
// float4 of the rank-wide row (rank <= 512).
__global__ void __launch_bounds__(256) combine_kernel(int batch, int q_len, int H, int rank, int max_kv, int S,
                                                     const int32_t *__restrict__ kv_len,
                                                     const float *__restrict__ o_part,
                                                     const float *__restrict__ lse_part, float *o_lat,
                                                     float *lse_out)
{
    __shared__ int64_t red[32];
    const int b = blockIdx.x;
    const int64_t T = block_tile_sum(kv_len, batch, q_len, max_kv, red);
    const int64_t t0 = block_tile_sum(kv_len, b, q_len, max_kv, red);
    const int64_t nb = seq_tiles(kv_len[b], q_len, max_kv);
    if (nb == 0 || T == 0) return;  // invalid length: recorded by the attention kernel
    const int k_first = part_of_tile(t0, T, S), k_last = part_of_tile(t0 + nb - 1, T, S);
    const int rows = q_len * H;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    const int nvec = rank / 4;
    for (int row = warp; row < rows; row += nwarps) {
        float m = -INFINITY;
        for (int k = k_first; k <= k_last; ++k) {
            if (part_begin(k, T, S) == part_begin(k + 1, T, S)) continue;  // empty partition
            m = fmaxf(m, lse_part[(static_cast<int64_t>(b) + k) * rows + row]);
        }
        float4 acc[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        float wsum = 0.f;
        if (m != -INFINITY) {
            for (int k = k_first; k <= k_last; ++k) {
                if (part_begin(k, T, S) == part_begin(k + 1, T, S)) continue;
                const int64_t slot = static_cast<int64_t>(b) + k;
                const float l = lse_part[slot * rows + row];
                if (l == -INFINITY) continue;
                const float w = __expf(l - m);
                wsum += w;
                const float4 *src = reinterpret_cast<const float4 *>(o_part + (slot * rows + row) * rank);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int v = lane + 32 * u;
                    if (v < nvec) {
                        const float4 x = src[v];
                        acc[u].x += w * x.x;
                        acc[u].y += w * x.y;
                        acc[u].z += w * x.z;
                        acc[u].w += w * x.w;
                    }
                }
            }
        }
        const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
        float4 *dst = reinterpret_cast<float4 *>(o_lat + (static_cast<int64_t>(b) * rows + row) * rank);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int v = lane + 32 * u;
            if (v < nvec) dst[v] = make_float4(acc[u].x * inv, acc[u].y * inv, acc[u].z * inv, acc[u].w * inv);
        }
        if (lse_out && lane == 0) lse_out[static_cast<int64_t>(b) * rows + row] = wsum > 0.f ? m + logf(wsum) : -INFINITY;
    }
}

}  // namespace

cudaError_t launch_combine(int batch, int q_len, int num_heads, int rank, int max_kv, int num_splits,
                           const int32_t *kv_len, const float *o_part, const float *lse_part, float *o_lat,
                           float *lse, cudaStream_t st)
{
    combine_kernel<<<batch, 256, 0, st>>>(batch, q_len, num_heads, rank, max_kv, num_splits, kv_len, o_part,
                                          lse_part, o_lat, lse);
    return cudaGetLastError();
}

}  // namespace gbmla
