// mla_absorb_q: latent query q_lat = W_UK[g]^T q_nope (attention "through
// absorbed projections", Sec. 1; Eq. 5 read right to left) and the positional
// query rotated to its own position (Sec. 3.1).
#include "common.cuh"
#include "internal.h"
#include "simt_gemm.cuh"

namespace gbmla {
namespace {

// Rows of group g: (bi, hh) with bi = b*q_len + i and head g*hpg + hh.
__global__ void __launch_bounds__(256) absorb_gemm_kernel(int rows_g, int H, int hpg, int d_nope, int rank,
                                                         int ld_out, const uint16_t *__restrict__ q_nope,
                                                         const uint16_t *__restrict__ w_uk, uint16_t *q_abs)
{
    const int g = blockIdx.z;
    auto grow = [=](int m) { return static_cast<int64_t>(m / hpg) * H + g * hpg + m % hpg; };
    const uint16_t *w = w_uk + static_cast<int64_t>(g) * d_nope * rank;
    simt_gemm_64x64(
        blockIdx.x * 64, blockIdx.y * 64, rows_g, rank, d_nope,
        [=](int m, int k) { return bf16_bits_to_float(q_nope[grow(m) * d_nope + k]); },
        [=](int n, int k) { return bf16_bits_to_float(w[static_cast<int64_t>(k) * rank + n]); },
        [=](int m, int n, float v) { q_abs[grow(m) * ld_out + n] = __bfloat16_as_ushort(__float2bfloat16_rn(v)); });
}

// One block per (b, i): angles of position kv_len[b] - q_len + i are shared
// by all heads.
__global__ void __launch_bounds__(256) absorb_rope_kernel(int q_len, int H, int rank, int d_rope, int style,
                                                         float base, const int32_t *__restrict__ kv_len,
                                                         const uint16_t *__restrict__ q_pe, uint16_t *q_abs)
{
    __shared__ float cs[64], sn[64];
    const int bi = blockIdx.x;
    const int b = bi / q_len, i = bi % q_len;
    const int half = d_rope / 2;
    const int64_t pos = static_cast<int64_t>(kv_len[b]) - q_len + i;
    for (int e = threadIdx.x; e < half; e += blockDim.x) rope_cos_sin(pos, rope_theta(e, d_rope, base), &cs[e], &sn[e]);
    __syncthreads();
    const int ld = rank + d_rope;
    for (int t = threadIdx.x; t < H * half; t += blockDim.x) {
        const int h = t / half, e = t % half;
        const int64_t row = static_cast<int64_t>(bi) * H + h;
        const int i0 = style == 0 ? e : 2 * e;
        const int i1 = style == 0 ? e + half : 2 * e + 1;
        const float x0 = bf16_bits_to_float(q_pe[row * d_rope + i0]);
        const float x1 = bf16_bits_to_float(q_pe[row * d_rope + i1]);
        q_abs[row * ld + rank + i0] = __bfloat16_as_ushort(__float2bfloat16_rn(x0 * cs[e] - x1 * sn[e]));
        q_abs[row * ld + rank + i1] = __bfloat16_as_ushort(__float2bfloat16_rn(x1 * cs[e] + x0 * sn[e]));
    }
}

}  // namespace

cudaError_t launch_absorb(const mla_dims &d, int batch, int q_len, const void *q_nope, const void *q_pe,
                          const int32_t *kv_len, const void *w_uk, void *q_abs, unsigned *status,
                          cudaStream_t st)
{
    (void)status;
    const int H = d.num_heads, G = d.num_kv_groups, hpg = H / G;
    const int rows_g = batch * q_len * hpg;
    dim3 grid((rows_g + 63) / 64, (d.rank + 63) / 64, G);
    absorb_gemm_kernel<<<grid, 256, 0, st>>>(rows_g, H, hpg, d.d_nope, d.rank, d.rank + d.d_rope,
                                             static_cast<const uint16_t *>(q_nope),
                                             static_cast<const uint16_t *>(w_uk), static_cast<uint16_t *>(q_abs));
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    absorb_rope_kernel<<<batch * q_len, 256, 0, st>>>(q_len, H, d.rank, d.d_rope, d.rope_style, d.rope_base, kv_len,
                                                      static_cast<const uint16_t *>(q_pe),
                                                      static_cast<uint16_t *>(q_abs));
    return cudaGetLastError();
}

}  // namespace gbmla
