// mla_out_proj: o = W_UV[g] o_lat (Eq. 5) and optionally out = W_O concat_h o
// (the block output "after its fixed output projection", Sec. 4.1).
#include "common.cuh"
#include "internal.h"
#include "simt_gemm.cuh"

namespace gbmla {
namespace {

__global__ void __launch_bounds__(256) up_proj_kernel(int rows_g, int H, int hpg, int rank, int d_v,
                                                     const float *__restrict__ o_lat,
                                                     const uint16_t *__restrict__ w_uv, uint16_t *o)
{
    const int g = blockIdx.z;
    auto grow = [=](int m) { return static_cast<int64_t>(m / hpg) * H + g * hpg + m % hpg; };
    const uint16_t *w = w_uv + static_cast<int64_t>(g) * d_v * rank;
    simt_gemm_64x64(
        blockIdx.x * 64, blockIdx.y * 64, rows_g, d_v, rank,
        [=](int m, int k) { return o_lat[grow(m) * rank + k]; },
        [=](int n, int k) { return bf16_bits_to_float(w[static_cast<int64_t>(n) * rank + k]); },
        [=](int m, int n, float v) { o[grow(m) * d_v + n] = __bfloat16_as_ushort(__float2bfloat16_rn(v)); });
}

__global__ void __launch_bounds__(256) o_proj_kernel(int rows, int hidden, int kdim,
                                                    const uint16_t *__restrict__ o,
                                                    const uint16_t *__restrict__ w_o, uint16_t *out)
{
    simt_gemm_64x64(
        blockIdx.x * 64, blockIdx.y * 64, rows, hidden, kdim,
        [=](int m, int k) { return bf16_bits_to_float(o[static_cast<int64_t>(m) * kdim + k]); },
        [=](int n, int k) { return bf16_bits_to_float(w_o[static_cast<int64_t>(n) * kdim + k]); },
        [=](int m, int n, float v) {
            out[static_cast<int64_t>(m) * hidden + n] = __bfloat16_as_ushort(__float2bfloat16_rn(v));
        });
}

}  // namespace

cudaError_t launch_out_proj(const mla_dims &d, int batch, int q_len, const float *o_lat, const void *w_uv,
                            const void *w_o, void *o, void *out, cudaStream_t st)
{
    const int H = d.num_heads, G = d.num_kv_groups, hpg = H / G;
    const int rows_g = batch * q_len * hpg;
    dim3 g1((rows_g + 63) / 64, (d.d_v + 63) / 64, G);
    up_proj_kernel<<<g1, 256, 0, st>>>(rows_g, H, hpg, d.rank, d.d_v, o_lat, static_cast<const uint16_t *>(w_uv),
                                       static_cast<uint16_t *>(o));
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || w_o == nullptr || d.hidden == 0) return e;
    const int rows = batch * q_len;
    dim3 g2((rows + 63) / 64, (d.hidden + 63) / 64);
    o_proj_kernel<<<g2, 256, 0, st>>>(rows, d.hidden, H * d.d_v, static_cast<const uint16_t *>(o),
                                      static_cast<const uint16_t *>(w_o), static_cast<uint16_t *>(out));
    return cudaGetLastError();
}

}  // namespace gbmla
