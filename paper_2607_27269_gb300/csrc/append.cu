// mla_cache_append: write this step's latent rows and RoPE-rotated positional
// keys into a contiguous or paged cache (Sec. 3.2 latent cache, Sec. 3.1 R_t).
#include "common.cuh"
#include "internal.h"

namespace gbmla {
namespace {

// One block per appended entry (k, b).  The latent row is a bit-exact 16-byte
// vector copy; the positional key is rotated in fp32 (angle reduced exactly
// as a fixed-point fraction of a turn) and rounded to bf16, nearest-even.
__global__ void __launch_bounds__(128) cache_append_kernel(CacheView c, int rank, int d_rope, int style,
                                                          const RopeTurns turns, int n_new,
                                                          const uint16_t *__restrict__ c_new,
                                                          const uint16_t *__restrict__ kr_new,
                                                          const int32_t *__restrict__ start_pos,
                                                          unsigned *status, int groups)
{
    // no early trigger: a cache writer lets its dependents launch only once it
    // has completed (the attention kernel loads cache tiles before its wait)
    griddep_wait();
    const int k = blockIdx.x, b = blockIdx.y;
    const int64_t pos = static_cast<int64_t>(start_pos[b / groups]) + k;
    if (pos < 0 || pos >= c.capacity) {
        if (threadIdx.x == 0) record_status(status, kStatusBounds);
        return;
    }
    int64_t blk, slot;
    if (c.block_table) {
        const int32_t page = c.block_table[static_cast<int64_t>(b) * c.bt_stride + pos / c.page_size];
        if (page < 0 || page >= c.num_pages) {
            if (threadIdx.x == 0) record_status(status, kStatusBounds);
            return;
        }
        blk = page;
        slot = pos % c.page_size;
    } else {
        blk = b;
        slot = pos;
    }
    uint16_t *crow = (uint16_t *)c.c_kv + blk * c.c_blk + slot * c.c_tok;
    uint16_t *rrow = (uint16_t *)c.k_rope + blk * c.r_blk + slot * c.r_tok;
    const int64_t entry = groups == 1 ? static_cast<int64_t>(b) * n_new + k
                                      : (static_cast<int64_t>(b / groups) * n_new + k) * groups + b % groups;
    const uint4 *src = reinterpret_cast<const uint4 *>(c_new + entry * rank);
    for (int v = threadIdx.x; v < rank / 8; v += blockDim.x) reinterpret_cast<uint4 *>(crow)[v] = src[v];

    const uint16_t *kr = kr_new + entry * d_rope;
    const int half = d_rope / 2;
    for (int e = threadIdx.x; e < half; e += blockDim.x) {
        float cs, sn;
        rope_cos_sin(pos, turns.f[e], &cs, &sn);
        const int i0 = style == 0 ? e : 2 * e;
        const int i1 = style == 0 ? e + half : 2 * e + 1;
        const float x0 = bf16_bits_to_float(kr[i0]), x1 = bf16_bits_to_float(kr[i1]);
        const float y0 = x0 * cs - x1 * sn;
        const float y1 = x1 * cs + x0 * sn;
        rrow[i0] = __bfloat16_as_ushort(__float2bfloat16_rn(y0));
        rrow[i1] = __bfloat16_as_ushort(__float2bfloat16_rn(y1));
    }
}

}  // namespace

cudaError_t launch_append(const mla_dims &d, const CacheView &c, int batch, int n_new, const void *c_new,
                          const void *kr_new, const int32_t *start_pos, unsigned *status, cudaStream_t st,
                          int groups)
{
    dim3 grid(n_new, batch);
    return launch_dependent(cache_append_kernel, grid, dim3(128), 0, st, 1, c, d.rank, d.d_rope, d.rope_style,
                            rope_turns(d.d_rope, d.rope_base), n_new, static_cast<const uint16_t *>(c_new),
                            static_cast<const uint16_t *>(kr_new), start_pos, status, groups);
}

}  // namespace gbmla
