// mla_combine: merge the split-KV partials of each sequence with their
// log-sum-exp weights (the softmax normaliser of Eq. 3).
#include <math.h>

#include "common.cuh"
#include "internal.h"

namespace gbmla {
namespace {

// Block (row group, sequence b).  A row of o_lat is rank floats; `tpr`
// threads share it, each owning VEC consecutive float4 (so tpr = rank / 4 /
// VEC), and a 256-thread block covers 256 / tpr rows.  Every partial of the
// row is read once, with all of them in flight at the same time.
template <int VEC>
__global__ void __launch_bounds__(256) combine_kernel(int batch, int q_len, int H, int rank, int max_kv, int S,
                                                     const int32_t *__restrict__ kv_len,
                                                     const float *__restrict__ o_part,
                                                     const float *__restrict__ lse_part, float *o_lat,
                                                     float *lse_out)
{
    griddep_wait();
    griddep_launch_dependents();
    __shared__ int64_t red[64];
    const int b = blockIdx.y;
    int64_t T, t0;
    block_tile_sums(kv_len, batch, b, q_len, max_kv, red, &T, &t0);
    const int64_t nb = seq_tiles(kv_len[b], q_len, max_kv);
    if (nb == 0 || T == 0) return;  // invalid length: recorded by the attention kernel
    const int k_first = part_of_tile(t0, T, S), k_last = part_of_tile(t0 + nb - 1, T, S);
    const int rows = q_len * H;
    const int tpr = rank / (4 * VEC);
    const int rpb = blockDim.x / tpr;
    const int row = blockIdx.x * rpb + threadIdx.x / tpr;
    const int part = threadIdx.x % tpr;
    if (row >= rows) return;
    // a partition is empty only when there are fewer tiles than partitions
    const bool may_be_empty = T < S;
    auto empty = [&](int k) { return may_be_empty && part_begin(k, T, S) == part_begin(k + 1, T, S); };
    // exponent base: the largest partial log-sum-exp of the row
    float m = -INFINITY;
    for (int k = k_first; k <= k_last; ++k) {
        if (empty(k)) continue;
        m = fmaxf(m, lse_part[(static_cast<int64_t>(b) + k) * rows + row]);
    }
    float4 acc[VEC];
#pragma unroll
    for (int u = 0; u < VEC; ++u) acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
    float wsum = 0.f;
    if (m != -INFINITY) {
        // four partitions per step, their loads issued together
        for (int k4 = k_first; k4 <= k_last; k4 += 4) {
            float wk[4];
            float4 x[4][VEC];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int k = k4 + j;
                wk[j] = 0.f;
                if (k <= k_last && !empty(k)) {
                    const int64_t slot = static_cast<int64_t>(b) + k;
                    const float l = lse_part[slot * rows + row];
                    if (l != -INFINITY) {
                        wk[j] = __expf(l - m);
                        const float4 *src =
                            reinterpret_cast<const float4 *>(o_part + (slot * rows + row) * rank) + part * VEC;
#pragma unroll
                        for (int u = 0; u < VEC; ++u) x[j][u] = __ldcs(src + u);  // read once: do not keep in L2
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                if (wk[j] == 0.f) continue;
                wsum += wk[j];
#pragma unroll
                for (int u = 0; u < VEC; ++u) {
                    acc[u].x += wk[j] * x[j][u].x;
                    acc[u].y += wk[j] * x[j][u].y;
                    acc[u].z += wk[j] * x[j][u].z;
                    acc[u].w += wk[j] * x[j][u].w;
                }
            }
        }
    }
    const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
    float4 *dst = reinterpret_cast<float4 *>(o_lat + (static_cast<int64_t>(b) * rows + row) * rank) + part * VEC;
#pragma unroll
    for (int u = 0; u < VEC; ++u) dst[u] = make_float4(acc[u].x * inv, acc[u].y * inv, acc[u].z * inv, acc[u].w * inv);
    if (lse_out && part == 0)
        lse_out[static_cast<int64_t>(b) * rows + row] = wsum > 0.f ? m + logf(wsum) : -INFINITY;
}

}  // namespace

cudaError_t launch_combine(int batch, int q_len, int num_heads, int rank, int max_kv, int num_splits,
                           const int32_t *kv_len, const float *o_part, const float *lse_part, float *o_lat,
                           float *lse, cudaStream_t st)
{
    // rank is a multiple of 64 (<= 512): 2 float4 per thread gives tpr = rank / 8 <= 64
    const int tpr = rank / 8, rpb = 256 / tpr;
    const int rows = q_len * num_heads;
    dim3 grid((rows + rpb - 1) / rpb, batch);
    if (batch == 0 || rows == 0) return cudaSuccess;
    return launch_dependent(combine_kernel<2>, grid, dim3(256), 0, st, 1, batch, q_len, num_heads, rank, max_kv,
                            num_splits, kv_len, o_part, lse_part, o_lat, lse);
}

}  // namespace gbmla
