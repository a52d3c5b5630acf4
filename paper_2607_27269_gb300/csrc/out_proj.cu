// mla_out_proj: o = W_UV[g] o_lat (Eq. 5) and optionally out = W_O concat_h o
// (the block output "after its fixed output projection", Sec. 4.1), both as
// grouped GEMMs.
#include "common.cuh"
#include "internal.h"

namespace gbmla {

cudaError_t launch_out_proj(const mla_dims &d, int batch, int q_len, const float *o_lat, const void *w_uv,
                            const void *w_o, void *o, void *out, unsigned *status, cudaStream_t st)
{
    const int H = d.num_heads, G = d.num_kv_groups, hpg = H / G;
    GroupGemm p;
    p.M = batch * q_len * hpg;  // rows (b, i, head g*hpg + hh) of group g
    p.N = d.d_v;
    p.K = d.rank;
    p.G = G;
    p.hpg = hpg;
    p.blk = H;
    p.A = o_lat;
    p.a_f32 = 1;
    p.lda = d.rank;
    p.B = w_uv;  // [G][d_v][rank]: K-major
    p.b_nmajor = 0;
    p.C = o;
    p.ldc = d.d_v;
    p.status = status;
    cudaError_t e = launch_group_gemm(p, st);
    if (e != cudaSuccess || w_o == nullptr || d.hidden == 0) return e;
    GroupGemm q;
    q.M = batch * q_len;
    q.N = d.hidden;
    q.K = H * d.d_v;
    q.G = 1;
    q.hpg = 1;
    q.blk = 1;
    q.A = o;
    q.a_f32 = 0;
    q.lda = H * d.d_v;
    q.B = w_o;  // [hidden][H d_v]: K-major
    q.b_nmajor = 0;
    q.C = out;
    q.ldc = d.hidden;
    q.status = status;
    return launch_group_gemm(q, st);
}

}  // namespace gbmla
