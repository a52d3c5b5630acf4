// mla_absorb_q: latent query q_lat = W_UK[g]^T q_nope (attention "through
// absorbed projections", Sec. 1; Eq. 5 read right to left) and the positional
// query rotated to its own position (Sec. 3.1).
#include "common.cuh"
#include "internal.h"

namespace gbmla {
namespace {

// One block per (b, i): angles of position kv_len[b] - q_len + i are shared
// by all heads.
__global__ void __launch_bounds__(256) absorb_rope_kernel(int q_len, int H, int rank, int d_rope, int style,
                                                         const RopeTurns turns, const int32_t *__restrict__ kv_len,
                                                         const uint16_t *__restrict__ q_pe, uint16_t *q_abs)
{
    griddep_wait();
    griddep_launch_dependents();
    __shared__ float cs[64], sn[64];
    const int bi = blockIdx.x;
    const int b = bi / q_len, i = bi % q_len;
    const int half = d_rope / 2;
    const int64_t pos = static_cast<int64_t>(kv_len[b]) - q_len + i;
    for (int e = threadIdx.x; e < half; e += blockDim.x) rope_cos_sin(pos, turns.f[e], &cs[e], &sn[e]);
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
    const int H = d.num_heads, G = d.num_kv_groups, hpg = H / G;
    // rows of group g: (b, i, head g*hpg + hh); q_lat = q_nope W_UK[g] (W_UK: d_nope x rank)
    GroupGemm p;
    p.M = batch * q_len * hpg;
    p.N = d.rank;
    p.K = d.d_nope;
    p.G = G;
    p.hpg = hpg;
    p.blk = H;
    p.A = q_nope;
    p.a_f32 = 0;
    p.lda = d.d_nope;
    p.B = w_uk;
    p.b_nmajor = 1;
    p.C = q_abs;
    p.ldc = d.rank + d.d_rope;
    p.status = status;
    cudaError_t e = launch_group_gemm(p, st);
    if (e != cudaSuccess) return e;
    return launch_dependent(absorb_rope_kernel, dim3(batch * q_len), dim3(256), 0, st, 1, q_len, H, d.rank, d.d_rope,
                            d.rope_style, rope_turns(d.d_rope, d.rope_base), kv_len, static_cast<const uint16_t *>(q_pe),
                            static_cast<uint16_t *>(q_abs));
}

}  // namespace gbmla
