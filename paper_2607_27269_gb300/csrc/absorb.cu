// mla_absorb_q: latent query q_lat = W_UK[g]^T q_nope (attention "through
// absorbed projections", Sec. 1; Eq. 5 read right to left) and the positional
// query rotated to its own position (Sec. 3.1).
#include "common.cuh"
#include "internal.h"

namespace gbmla {

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
    // one launch: the GEMM's first column tile also rotates the positional query
    return launch_absorb_gemm(p, d, q_pe, kv_len, q_len, st);
}

}  // namespace gbmla
