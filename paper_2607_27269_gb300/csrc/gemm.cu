// The projections of the decode step as grouped GEMMs (all bf16 weights,
// fp32 accumulation, bf16 results):
//   absorption (Sec. 1; Eq. 5 read right to left): q_lat[row] = q_nope[row] W_UK[g]   (W_UK: d_nope x r)
//   value up-projection (Eq. 5):                    o[row]     = W_UV[g] o_lat[row]    (W_UV: d_v x r)
//   output projection (Sec. 4.1):                   out[m]     = W_O concat_h o[m]     (W_O: D x H d_v)
// In every case C[phys(g, m), n] = sum_k A[phys(g, m), k] B_g(n, k) for the M
// rows of group g, with phys(g, m) = (m / hpg) * blk + g * hpg + m % hpg.
//
// All as one tcgen05 GEMM: up to 128 rows x BN columns per CTA, A and the
// weight tile loaded by TMA, the fp32 accumulator in TMEM.  A GEMM whose tiles
// would occupy few SMs (few rows, deep K: the output projection of a small
// batch) splits K over a cluster of up to four CTAs; each leaves its partial
// tile in shared memory and the cluster sums the partials in a fixed order
// through distributed shared memory, so the result does not depend on timing.
//
// The same kernel, with PROJ set, projects the step's hidden states (the step
// before the cache append, Sec. 3.2 and Eq. 1): rows are the entries
// h[b, k, :], and the column tiles run over W^DKV (the latent), one tile for
// W^KR (the positional key) and W^Q (the queries).  Its epilogue writes the
// latent row and the positional key, rotated to the entry's position in fp32,
// straight into the (paged) cache, and splits each query head into its
// non-positional and positional parts.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace gbmla {
namespace {

__device__ __forceinline__ int64_t phys_row(const GroupGemm &p, int g, int m)
{
    return static_cast<int64_t>(m / p.hpg) * p.blk + g * p.hpg + m % p.hpg;
}

// Epilogue arguments of the projection (PROJ): column tiles [0, tiles_lat)
// hold the latent, tile tiles_lat the positional key, the rest the queries.
// The absorption GEMM (not PROJ) reuses it for the positional query: when
// rope_src is set, the CTAs of each row tile also write
// C[row, rank .. rank + d_rope) = R_p q_pe[row] for the rows of that tile,
// p = kv_len[b] - q_len + i for row (b, i, head) (rows in [B, q_len, heads] order).
struct ProjEpi {
    CacheView cache;
    const int32_t *start_pos;
    uint16_t *q_nope, *q_pe;
    int n_new, rank, d_rope, d_nope, heads, style;
    RopeTurns turns;
    int tiles_lat;
    uint32_t box_bytes[3];  // weight-tile bytes of the three column regions
    const uint16_t *rope_src;  // absorption: q_pe [B, q_len, heads, d_rope], or null
    const int32_t *kv_len;
    int q_len;
};

__device__ __forceinline__ void store16_bf16(uint16_t *dst, const uint32_t (&v)[16])
{
    uint32_t w[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const __nv_bfloat162 b = __floats2bfloat162_rn(__uint_as_float(v[2 * e]), __uint_as_float(v[2 * e + 1]));
        w[e] = *reinterpret_cast<const uint32_t *>(&b);
    }
    reinterpret_cast<uint4 *>(dst)[0] = make_uint4(w[0], w[1], w[2], w[3]);
    reinterpret_cast<uint4 *>(dst)[1] = make_uint4(w[4], w[5], w[6], w[7]);
}

// R_pos of the DR projected positional-key values x (fp32; the angle reduced
// exactly as a fraction of a turn), rounded once to bf16 into `row`.
template <int DR>
__device__ __forceinline__ void rotate_store(const float (&x)[64], int64_t pos, int style, const RopeTurns &turns,
                                             uint16_t *row)
{
    constexpr int HALF = DR / 2;
    __align__(16) uint16_t y[DR];
    if (style == 0) {
#pragma unroll
        for (int k = 0; k < HALF; ++k) {
            float cs, sn;
            rope_cos_sin(pos, turns.f[k], &cs, &sn);
            y[k] = __bfloat16_as_ushort(__float2bfloat16_rn(x[k] * cs - x[k + HALF] * sn));
            y[k + HALF] = __bfloat16_as_ushort(__float2bfloat16_rn(x[k + HALF] * cs + x[k] * sn));
        }
    } else {
#pragma unroll
        for (int k = 0; k < HALF; ++k) {
            float cs, sn;
            rope_cos_sin(pos, turns.f[k], &cs, &sn);
            y[2 * k] = __bfloat16_as_ushort(__float2bfloat16_rn(x[2 * k] * cs - x[2 * k + 1] * sn));
            y[2 * k + 1] = __bfloat16_as_ushort(__float2bfloat16_rn(x[2 * k + 1] * cs + x[2 * k] * sn));
        }
    }
#pragma unroll
    for (int v = 0; v < DR / 8; ++v) reinterpret_cast<uint4 *>(row)[v] = reinterpret_cast<const uint4 *>(y)[v];
}

// Projection epilogue for tile row m (the entry h[m / n_new, m % n_new]);
// every lane of the warp calls it (the TMEM loads are warp-collective).
template <int BN>
__device__ void proj_epilogue(const GroupGemm &p, const ProjEpi &e, uint32_t t_lane, int m, bool row_ok)
{
    const int ty = blockIdx.y;
    if (ty > e.tiles_lat) {
        // ---- queries: column c of W^Q is element c % dq of head c / dq
        const int dq = e.d_nope + e.d_rope, nq = e.heads * dq;
        const int c0 = (ty - e.tiles_lat - 1) * BN;
#pragma unroll 1
        for (int j = 0; j < BN; j += 16) {
            uint32_t v[16];
            tc::ld_32x32b_x16(t_lane + j, v);
            tc::wait_ld();
            const int c = c0 + j;
            if (!row_ok || c >= nq) continue;
            const int head = c / dq, el = c % dq;
            const int64_t hrow = static_cast<int64_t>(m) * e.heads + head;
            if (c + 16 <= nq && el + 16 <= e.d_nope) {
                store16_bf16(e.q_nope + hrow * e.d_nope + el, v);
            } else if (c + 16 <= nq && el >= e.d_nope && el + 16 <= dq) {
                store16_bf16(e.q_pe + hrow * e.d_rope + (el - e.d_nope), v);
            } else {
                for (int u = 0; u < 16 && c + u < nq; ++u) {
                    const int hu = (c + u) / dq, eu = (c + u) % dq;
                    const int64_t r = static_cast<int64_t>(m) * e.heads + hu;
                    const uint16_t b = __bfloat16_as_ushort(__float2bfloat16_rn(__uint_as_float(v[u])));
                    if (eu < e.d_nope)
                        e.q_nope[r * e.d_nope + eu] = b;
                    else
                        e.q_pe[r * e.d_rope + (eu - e.d_nope)] = b;
                }
            }
        }
        return;
    }
    // ---- the entry's cache row: position start_pos[b] + k, through the block table when paged
    const CacheView &c = e.cache;
    bool ok = row_ok;
    int64_t pos = 0, blk = 0, slot = 0;
    if (ok) {
        const int b = m / e.n_new, k = m % e.n_new;
        pos = static_cast<int64_t>(e.start_pos[b]) + k;
        ok = pos >= 0 && pos < c.capacity;
        if (ok && c.block_table) {
            const int32_t page = c.block_table[static_cast<int64_t>(b) * c.bt_stride + pos / c.page_size];
            ok = page >= 0 && page < c.num_pages;
            blk = page;
            slot = pos % c.page_size;
        } else {
            blk = b;
            slot = pos;
        }
        if (!ok) record_status(p.status, kStatusBounds);
    }
    if (ty < e.tiles_lat) {
        // ---- latent c = W^DKV h, rounded once
        uint16_t *crow = static_cast<uint16_t *>(const_cast<void *>(c.c_kv)) + blk * c.c_blk + slot * c.c_tok;
#pragma unroll 1
        for (int j = 0; j < BN; j += 16) {
            uint32_t v[16];
            tc::ld_32x32b_x16(t_lane + j, v);
            tc::wait_ld();
            if (ok) store16_bf16(crow + ty * BN + j, v);
        }
        return;
    }
    // ---- positional key R_pos W^KR h (d_rope = 32 or 64 columns of this tile)
    float x[64];
#pragma unroll
    for (int j = 0; j < 64; j += 16) {
        if (j < e.d_rope) {
            uint32_t v[16];
            tc::ld_32x32b_x16(t_lane + j, v);
            tc::wait_ld();
#pragma unroll
            for (int u = 0; u < 16; ++u) x[j + u] = __uint_as_float(v[u]);
        } else {
#pragma unroll
            for (int u = 0; u < 16; ++u) x[j + u] = 0.f;
        }
    }
    if (!ok) return;
    uint16_t *rrow = static_cast<uint16_t *>(const_cast<void *>(c.k_rope)) + blk * c.r_blk + slot * c.r_tok;
    if (e.d_rope == 64)
        rotate_store<64>(x, pos, e.style, e.turns, rrow);
    else
        rotate_store<32>(x, pos, e.style, e.turns, rrow);
}

// ---------------------------------------------------------------- tensor-core GEMM
// Both operands arrive by TMA.  The A rows of a group are one 4-d box
// (K, head in group, group, row block): a tile holds R = 128 / hpg row blocks
// of hpg rows, i.e. RT = R hpg <= 128 rows.  A bf16 A box lands directly in
// the 128B-swizzled K-major layout the MMA reads; an fp32 A (o_lat) lands as
// two 32-column boxes in a staging tile, which four warps convert to bf16.
constexpr int kStages = 16;  // most ring stages; fewer when K is short or shared memory runs out
constexpr int kGemmThreads = 192;  // warp 0 TMA, warp 1 MMA, warps 2..5 convert / epilogue

struct __align__(8) GemmBars {
    uint64_t full[kStages], raw_full[kStages], conv_done[kStages], empty[kStages], done;
};

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *map, int32_t c0, int32_t c1, int32_t c2,
                                            int32_t c3, uint32_t mbar)
{
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], "
        "[%6];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(mbar)
        : "memory");
}

// BN: columns per CTA.  NMAJ: the weight is N-major.  AF32: A is fp32.
// PROJ: the projection (K-major weights map_b, map_b2, map_b3 by column region).
template <int BN, bool NMAJ, bool AF32, bool PROJ>
__global__ void __launch_bounds__(kGemmThreads) gemm_tc_kernel(const __grid_constant__ GroupGemm p,
                                                               const __grid_constant__ CUtensorMap map_a,
                                                               const __grid_constant__ CUtensorMap map_b,
                                                               const __grid_constant__ CUtensorMap map_b2,
                                                               const __grid_constant__ CUtensorMap map_b3,
                                                               const __grid_constant__ ProjEpi pe)
{
    static_assert(!PROJ || (!NMAJ && !AF32), "the projection reads bf16 h and K-major weights");
    constexpr int kABytes = 128 * 128;     // 128 rows x 64 K, bf16, SW128 K-major
    constexpr int kRawBytes = AF32 ? 2 * 128 * 128 : 0;  // two 32-column fp32 boxes
    constexpr int kBBytes = BN * 128;      // BN x 64 K (K-major) or 64 K x BN (N-major)
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ GemmBars bars;
    __shared__ uint32_t tmem_base;
    __shared__ int fail;
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~static_cast<uintptr_t>(1023));
    const int nk = (p.K + 63) / 64;
    const int ks = PROJ ? 1 : p.ksplit;                  // CTAs of the cluster sharing the K range
    const int kz = blockIdx.x % ks;                      // this CTA's share: chunks [c_begin, c_end)
    const int c_begin = kz * nk / ks, nkl = (kz + 1) * nk / ks - c_begin;
    const int NS = p.stages;                             // ring stages (<= kStages)
    // A stages sit a_stride apart: a full tile, or for a bf16 A of RT <= 64
    // rows just those rows (rounded to 8).  The M = 128 MMA still reads 128
    // rows from its stage base: the rows past RT come from the next stages or
    // the B ring (inside the allocation), land in accumulator rows >= RT and
    // are never stored.
    // An fp32 A has no A stages of its own: each converter thread writes its
    // bf16 row over the first half of its raw fp32 row, which it has read
    // before (chunk j of the row is written after the step that read it), so
    // a stage's bf16 tile is the first 16 KB of its raw stage.
    const int AS = AF32 ? 0 : PROJ ? kABytes : p.a_stride;
    unsigned char *sa = smem;                            // NS x A tile (bf16 A)
    unsigned char *sb = sa + NS * AS;                    // NS x B tile
    unsigned char *sr = sb + NS * kBBytes;               // NS x raw fp32 A, then its bf16 tile (AF32)
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int R = p.rblk, RT = R * p.hpg;                // row blocks and rows per tile (<= 128)
    const int mt = blockIdx.x / ks, n0 = blockIdx.y * BN, g = blockIdx.z;
    const int m0 = mt * RT;
    const uint32_t a_bytes = static_cast<uint32_t>(RT) * 128;  // per 64-column (bf16) or 32-column (fp32) box
    const uint64_t lim = kWaitLimitNs;

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&bars.full[s], 1);
            mbar_init(&bars.raw_full[s], 1);
            mbar_init(&bars.conv_done[s], 4);
            mbar_init(&bars.empty[s], 1);
        }
        mbar_init(&bars.done, 1);
        fail = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(smem_u32(&tmem_base), BN < 32 ? 32 : BN);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    griddep_wait();  // the activations come from the previous launch
    // the projection writes the cache: its dependents launch only once it has
    // completed (the attention kernel loads cache tiles before its own wait)
    if (!PROJ) griddep_launch_dependents();
    const uint32_t tmem = tmem_base;
    auto bail = [&]() {
        record_status(p.status, kStatusTimeout);
        fail = 1;
    };
    bool ep_ok = false;  // split K: this epilogue thread saw its CTA's MMAs complete

    if (warp == 0) {
        // ---- A and weight tiles by TMA
        const CUtensorMap *mb = &map_b;
        int brow = g * p.N + n0;
        uint32_t bbytes = kBBytes;
        if (PROJ) {
            const int ty = blockIdx.y, region = ty < pe.tiles_lat ? 0 : ty == pe.tiles_lat ? 1 : 2;
            mb = region == 0 ? &map_b : region == 1 ? &map_b2 : &map_b3;
            brow = region == 0 ? n0 : region == 1 ? 0 : (ty - pe.tiles_lat - 1) * BN;
            bbytes = pe.box_bytes[region];
        }
        if (lane == 0) {
            tc::prefetch_tensormap(&map_a);
            tc::prefetch_tensormap(mb);
        }
        for (int cc = 0; cc < nkl; ++cc) {
            const int c = c_begin + cc, s = cc % NS, round = cc / NS;
            if (round >= 1 && !__all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.empty[s]), (round - 1) & 1, lim))) {
                if (lane == 0) bail();
                break;
            }
            if (lane == 0) {
                const uint32_t fb = smem_u32(&bars.full[s]);
                tc::mbar_arrive_expect_tx(fb, bbytes + (AF32 ? 0u : a_bytes));
                const uint32_t dst = smem_u32(sb + s * kBBytes);
                if (NMAJ) {
                    // rows = K of group g, columns = N: one 64 x 64 box per 64 columns
                    for (int j = 0; j < BN / 64; ++j)
                        tc::tma_load_2d(dst + j * 64 * 128, &map_b, n0 + 64 * j, g * p.K + 64 * c, fb);
                } else {
                    tc::tma_load_2d(dst, mb, 64 * c, brow, fb);
                }
                if (AF32) {
                    const uint32_t rb = smem_u32(&bars.raw_full[s]);
                    tc::mbar_arrive_expect_tx(rb, 2 * a_bytes);
                    const uint32_t rdst = smem_u32(sr + s * kRawBytes);
                    tma_load_4d(rdst, &map_a, 64 * c, 0, g, mt * R, rb);
                    tma_load_4d(rdst + 128 * 128, &map_a, 64 * c + 32, 0, g, mt * R, rb);
                } else {
                    tma_load_4d(smem_u32(sa + s * AS), &map_a, 64 * c, 0, g, mt * R, fb);
                }
            }
            __syncwarp();
        }
    } else if (warp == 1) {
        // ---- MMA issuer (converged warp, one elected lane issues)
        const uint32_t idesc = tc::idesc_bf16_f32(128, BN, false, NMAJ);
        const uint64_t da = tc::smem_desc(0, 16, 1024, tc::kSwizzle128B);
        const uint64_t db = NMAJ ? tc::smem_desc(0, 64 * 128, 1024, tc::kSwizzle128B)
                                 : tc::smem_desc(0, 16, 1024, tc::kSwizzle128B);
        auto with_addr = [](uint64_t tmpl, uint32_t saddr) {
            return tmpl | static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
        };
        bool ok = true;
        for (int cc = 0; cc < nkl && ok; ++cc) {
            const int s = cc % NS, par = (cc / NS) & 1;
            ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.full[s]), par, lim) &&
                                             (!AF32 || mbar_wait(smem_u32(&bars.conv_done[s]), par, lim)));
            if (!ok) break;
            tc::fence_after_sync();
            const uint32_t a_base = smem_u32(AF32 ? sr + s * kRawBytes : sa + s * AS), b_base = smem_u32(sb + s * kBBytes);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
                const uint32_t b_addr = NMAJ ? b_base + kk * 16 * 128 : b_base + kk * 32;
                tc::mma_bf16_elect(tmem, with_addr(da, a_base + kk * 32), with_addr(db, b_addr), idesc,
                                   (cc | kk) != 0);
            }
            tc::commit_elect(smem_u32(&bars.empty[s]));
        }
        if (!ok && lane == 0) bail();
        tc::commit_elect(smem_u32(&bars.done));
    } else {
        if (AF32) {
            // ---- fp32 -> bf16: thread r converts tile row r (two 128-byte swizzled fp32 rows)
            const int r = tid - 64;
            for (int cc = 0; cc < nkl; ++cc) {
                const int s = cc % NS, par = (cc / NS) & 1;
                if (!__all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.raw_full[s]), par, lim))) {
                    if (lane == 0) bail();
                    break;
                }
                const uint4 *src0 = reinterpret_cast<const uint4 *>(sr + s * kRawBytes + r * 128);
                const uint4 *src1 = reinterpret_cast<const uint4 *>(sr + s * kRawBytes + 128 * 128 + r * 128);
                uint4 *dst = reinterpret_cast<uint4 *>(sr + s * kRawBytes + r * 128);  // over src0, in place
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    // bf16 16-byte chunk j = fp32 chunks 2j, 2j + 1 (of box j / 4)
                    const uint4 *src = j < 4 ? src0 : src1;
                    const int q0 = (2 * j) & 7, q1 = (2 * j + 1) & 7;
                    const float4 x = *reinterpret_cast<const float4 *>(&src[q0 ^ (r & 7)]);
                    const float4 y = *reinterpret_cast<const float4 *>(&src[q1 ^ (r & 7)]);
                    const __nv_bfloat162 b0 = __floats2bfloat162_rn(x.x, x.y), b1 = __floats2bfloat162_rn(x.z, x.w);
                    const __nv_bfloat162 b2 = __floats2bfloat162_rn(y.x, y.y), b3 = __floats2bfloat162_rn(y.z, y.w);
                    dst[j ^ (r & 7)] =
                        make_uint4(*reinterpret_cast<const uint32_t *>(&b0), *reinterpret_cast<const uint32_t *>(&b1),
                                   *reinterpret_cast<const uint32_t *>(&b2), *reinterpret_cast<const uint32_t *>(&b3));
                }
                tc::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(smem_u32(&bars.conv_done[s]));
            }
        }
        if (!PROJ && pe.rope_src) {
            // ---- the absorption's positional query, while the MMAs run.  The
            // tile's rows are whole (b, i) blocks of hpg heads (row m of group g
            // is head g hpg + m % hpg of token m / hpg), which share one
            // position: an item is one (token, pair) with one angle, applied to
            // the pair of every head of the group.  The items of this row tile
            // are spread over the CTAs that share it (column tiles, K shares).
            const int half = pe.d_rope / 2, hpg = p.hpg;
            const int slots = static_cast<int>(gridDim.y) * ks, slot = static_cast<int>(blockIdx.y) * ks + kz;
            const int tok0 = m0 / hpg, items = (min(RT, p.M - m0) / hpg) * half;
            // pair k: elements (k, k + half) in the half-split style, (2k, 2k + 1) interleaved
            const int s0 = pe.style == 0 ? 1 : 2, o1 = pe.style == 0 ? half : 1;
            for (int it = slot * 128 + (warp & 3) * 32 + lane; it < items; it += slots * 128) {
                const int k = it % half, bi = tok0 + it / half;  // bi = b q_len + i
                const int b = bi / pe.q_len, i = bi - b * pe.q_len;
                float cs, sn;
                rope_cos_sin(static_cast<int64_t>(__ldg(pe.kv_len + b)) - pe.q_len + i, pe.turns.f[k], &cs, &sn);
                const int64_t row0 = static_cast<int64_t>(bi) * p.blk + static_cast<int64_t>(g) * hpg;
                const int c0 = s0 * k, c1 = o1 + s0 * k;
                for (int h0 = 0; h0 < hpg; h0 += 4) {
                    uint16_t x0[4], x1[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        if (h0 + u < hpg) {
                            const uint16_t *src = pe.rope_src + (row0 + h0 + u) * pe.d_rope;
                            x0[u] = __ldg(src + c0);
                            x1[u] = __ldg(src + c1);
                        }
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        if (h0 + u < hpg) {
                            const float a0 = __uint_as_float(static_cast<uint32_t>(x0[u]) << 16);
                            const float a1 = __uint_as_float(static_cast<uint32_t>(x1[u]) << 16);
                            uint16_t *dst = static_cast<uint16_t *>(p.C) + (row0 + h0 + u) * p.ldc + pe.rank;
                            dst[c0] = __bfloat16_as_ushort(__float2bfloat16_rn(a0 * cs - a1 * sn));
                            dst[c1] = __bfloat16_as_ushort(__float2bfloat16_rn(a1 * cs + a0 * sn));
                        }
                }
            }
        }
        // ---- epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31
        const bool ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.done), 0, lim));
        if (!ok) {
            if (lane == 0) bail();
        } else if (!fail) {
            tc::fence_after_sync();
            const int q = warp & 3;
            const int i = q * 32 + lane;  // tile row
            const int me = m0 + i;
            const bool row_ok = i < RT && me < p.M;
            const uint32_t t_lane = tmem + (static_cast<uint32_t>(q * 32) << 16);
            const int64_t orow = row_ok ? phys_row(p, g, me) : 0;
            if (PROJ) {
                proj_epilogue<BN>(p, pe, t_lane, me, row_ok);
            } else if (ks > 1) {
                ep_ok = true;  // the partial is pushed once the whole cluster is past its MMAs
            } else {
#pragma unroll 1
            for (int j = 0; j < BN; j += 16) {
                uint32_t v[16];
                tc::ld_32x32b_x16(t_lane + j, v);
                tc::wait_ld();
                const int n = n0 + j;
                if (!row_ok || n >= p.N) continue;
                uint16_t *dst = static_cast<uint16_t *>(p.C) + orow * p.ldc + n;
                if (n + 16 <= p.N) {
                    store16_bf16(dst, v);
                } else {
                    for (int e = 0; e < 16 && n + e < p.N; ++e)
                        dst[e] = __bfloat16_as_ushort(__float2bfloat16_rn(__uint_as_float(v[e])));
                }
            }
            }
        }
    }
    if (!PROJ && ks > 1) {
        // (1) every CTA of the cluster is past its MMAs, so every ring is free;
        // (2) push this CTA's partial of each column slice to the slice's owner:
        // CTA o owns columns [o cw, (o + 1) cw) and receives, in its ring,
        // recv[r][row][cw + 4] from every rank r; (3) each owner sums its slice
        // in rank order (four columns per step) and stores the bf16 result
        const int cw = BN / ks;
        tc::cluster_sync();
        if (warp >= 2 && ep_ok && !fail) {
            tc::fence_after_sync();
            const int q = warp & 3, i = q * 32 + lane;
            const uint32_t t_lane = tmem + (static_cast<uint32_t>(q * 32) << 16);
            const uint32_t recv = smem_u32(smem);
#pragma unroll 1
            for (int j = 0; j < BN; j += 16) {
                uint32_t v[16];
                tc::ld_32x32b_x16(t_lane + j, v);
                tc::wait_ld();
                if (i < RT) {
                    const int o = j / cw;
                    const uint32_t local = recv + static_cast<uint32_t>(((kz * RT + i) * (cw + 4) + (j - o * cw)) * 4);
                    uint32_t remote;
                    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(o));
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote + 16 * e),
                                     "f"(__uint_as_float(v[4 * e])), "f"(__uint_as_float(v[4 * e + 1])),
                                     "f"(__uint_as_float(v[4 * e + 2])), "f"(__uint_as_float(v[4 * e + 3]))
                                     : "memory");
                }
            }
        }
        tc::cluster_sync();
        if (warp >= 2 && !fail) {
            const int q4 = cw / 4;
            const float *recv = reinterpret_cast<const float *>(smem);
            for (int idx = tid - 64; idx < RT * q4; idx += 128) {
                const int i = idx / q4, c4 = (idx % q4) * 4;
                const int me = m0 + i, n = n0 + kz * cw + c4;
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
                for (int r = 0; r < ks; ++r) {
                    const float4 v = *reinterpret_cast<const float4 *>(recv + (r * RT + i) * (cw + 4) + c4);
                    acc.x += v.x;
                    acc.y += v.y;
                    acc.z += v.z;
                    acc.w += v.w;
                }
                if (me >= p.M) continue;
                uint16_t *dst = static_cast<uint16_t *>(p.C) + phys_row(p, g, me) * p.ldc + n;
                const float a[4] = {acc.x, acc.y, acc.z, acc.w};
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (n + e < p.N) dst[e] = __bfloat16_as_ushort(__float2bfloat16_rn(a[e]));
            }
        }
        tc::cluster_sync();  // keep the cluster together until every CTA is done
    }
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, BN < 32 ? 32 : BN);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode_gemm = nullptr;

cudaError_t get_encoder()
{
    if (g_encode_gemm) return cudaSuccess;
    cudaDriverEntryPointQueryResult q;
    void *fn = nullptr;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return e != cudaSuccess ? e : cudaErrorNotSupported;
    g_encode_gemm = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return cudaSuccess;
}

// A: (K, head in group, group, row block) with the row mapping's strides.
bool encode_a(const GroupGemm &p, int rblk, bool f32, CUtensorMap *ma)
{
    const int es = f32 ? 4 : 2;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(p.K), static_cast<cuuint64_t>(p.hpg), static_cast<cuuint64_t>(p.G),
                          static_cast<cuuint64_t>(p.M / p.hpg)};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(p.lda) * es, static_cast<cuuint64_t>(p.hpg) * p.lda * es,
                             static_cast<cuuint64_t>(p.blk) * p.lda * es};
    cuuint32_t box[4] = {f32 ? 32u : 64u, static_cast<cuuint32_t>(p.hpg), 1u, static_cast<cuuint32_t>(rblk)};
    cuuint32_t es4[4] = {1, 1, 1, 1};
    return g_encode_gemm(ma, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4,
                         const_cast<void *>(p.A), dims, strides, box, es4, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// A K-major weight [rows][K] in boxes of 64 K x box_rows rows.
bool encode_kmajor(const void *w, int64_t rows, int K, int box_rows, CUtensorMap *mb)
{
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
    cuuint32_t box[2] = {64u, static_cast<cuuint32_t>(box_rows)}, es2[2] = {1, 1};
    return g_encode_gemm(mb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(w), dims, strides, box, es2,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Row blocks per tile: as many as fit 128 rows, but no more than there are
// (a short A box leaves the tile's other rows stale; their results are dropped).
int rows_per_tile(const GroupGemm &p) { return (128 / p.hpg) < (p.M / p.hpg) ? (128 / p.hpg) : (p.M / p.hpg); }

// Ring depth: as many stages as fit 192 KB, at most kStages and the K chunks.
template <int BN, bool AF32>
int ring_stages(int K, size_t *smem)
{
    const int nk = (K + 63) / 64;
    const size_t per_stage = (AF32 ? 2 * 128 * 128 : 128 * 128) + BN * 128;  // fp32 A: raw stage, bf16 in place
    int ns = static_cast<int>((192 * 1024) / per_stage);
    if (ns > kStages) ns = kStages;
    if (ns > nk) ns = nk;
    if (ns < 1) ns = 1;
    *smem = 1024 + static_cast<size_t>(ns) * per_stage;
    return ns;
}

template <int BN, bool NMAJ, bool AF32>
cudaError_t launch_tc(const GroupGemm &p, cudaStream_t st, const ProjEpi *rope = nullptr)
{
    cudaError_t e = get_encoder();
    if (e != cudaSuccess) return e;
    if (p.hpg < 1 || p.hpg > 128 || p.M % p.hpg) return cudaErrorInvalidValue;
    int rblk = rows_per_tile(p);
    const int ntiles = (p.N + BN - 1) / BN;
    const int nk = (p.K + 63) / 64;
    auto tiles_for = [&](int rb) { return static_cast<int64_t>((p.M / p.hpg + rb - 1) / rb) * ntiles * p.G; };
    // A grid too small to spread over the SMs and K too short to split (the
    // split below wants deep K): shorter row tiles instead, each CTA
    // re-reading its (small) weight tile from L2
    if (nk < 8)
        while (tiles_for(rblk) < 64 && rblk > 1 && rblk * p.hpg > 16) rblk = (rblk + 1) / 2;
    CUtensorMap ma, mb;
    if (!encode_a(p, rblk, AF32, &ma)) return cudaErrorInvalidValue;
    if (NMAJ) {  // [G K rows][N columns], 64 x 64 boxes
        cuuint64_t dims[2] = {static_cast<cuuint64_t>(p.N), static_cast<cuuint64_t>(p.G) * p.K};
        cuuint64_t strides[1] = {static_cast<cuuint64_t>(p.N) * 2};
        cuuint32_t box[2] = {64u, 64u}, es2[2] = {1, 1};
        CUresult r = g_encode_gemm(&mb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(p.B), dims, strides,
                                   box, es2, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    } else if (!encode_kmajor(p.B, static_cast<int64_t>(p.G) * p.N, p.K, BN, &mb)) {  // [G N rows][K columns]
        return cudaErrorInvalidValue;
    }
    const int rt = rblk * p.hpg;
    const int mtiles = (p.M + rt - 1) / rt;
    // Split K over a cluster when the tiles are short (<= 64 rows: a small
    // batch), K is deep (>= 8 chunks) and the tiles alone would leave most SMs
    // idle: up to 4 ways, at least two chunks each, with a ring of at most 4
    // stages so that two CTAs share an SM and the split grid runs in one wave.
    const int64_t tiles = static_cast<int64_t>(mtiles) * ntiles * p.G;
    int ks = 1;
    if (rt <= 64 && nk >= 8)
        while (ks < 4 && tiles * ks * 2 <= (AF32 ? 152 : 2 * 152) && nk >= 4 * ks) ks *= 2;  // fp32 A: one CTA per SM
    // Full 128-row tiles that would fill fewer than half the SMs (a mid-size
    // batch against a wide weight): split K as well, one CTA per SM, at least
    // eight chunks per share, the partials (128 rows x BN / ks columns from
    // each rank) pushed into the ring.  (Not for an fp32 A: there the
    // reduction cost as much as the split saved.)
    const bool wide_split = rt > 64 && !AF32 && nk >= 16 && tiles * 2 <= 152;
    if (wide_split)
        while (ks < 4 && tiles * ks * 2 <= 152 && nk >= 8 * ks) ks *= 2;
    size_t smem = 0;
    GroupGemm q = p;
    q.a_stride = 128 * 128;
    if (!AF32 && rt <= 64) {
        // short bf16 A tiles: stages of RT rows (rounded to 8), so that the ring
        // holds many more weight chunks -- with a split, all of a CTA's chunks
        // at two CTAs per SM -- and the weights stream with more bytes in flight
        q.a_stride = (rt + 7) / 8 * 8 * 128;
        const int nkl = (nk + ks - 1) / ks;
        const size_t per_stage = static_cast<size_t>(q.a_stride) + BN * 128;
        const size_t budget = ks > 1 ? 110 * 1024 : 192 * 1024;
        int ns = static_cast<int>(budget / per_stage);
        ns = ns > kStages ? kStages : ns;
        ns = ns > nkl ? nkl : ns;
        q.stages = ns < 1 ? 1 : ns;
        // the last stage's MMA reads a full 128-row window from its base
        const size_t ring = static_cast<size_t>(q.stages) * per_stage;
        const size_t window = static_cast<size_t>(q.stages - 1) * q.a_stride + 128 * 128;
        smem = 1024 + (ring > window ? ring : window);
    } else {
        q.stages = ring_stages<BN, AF32>((nk + ks - 1) / ks * 64, &smem);
        const size_t per_stage = (AF32 ? 2 * 128 * 128 : 128 * 128) + BN * 128;
        if (ks > 1 && !wide_split && q.stages > 4) {
            q.stages = 4;
            smem = 1024 + 4 * per_stage;
        }
        // an fp32-A grid just past one CTA per SM (W_UV of a large batch):
        // two stages, so that two CTAs share an SM and the grid runs in one wave
        if (AF32 && ks == 1 && tiles > 152 && tiles <= 2 * 152 && q.stages > 2) {
            q.stages = 2;
            smem = 1024 + 2 * per_stage;
        }
    }
    q.rblk = rblk;
    q.ksplit = ks;
    if (ks > 1) {  // the partials received from the cluster reuse the ring
        const size_t need = 1024 + static_cast<size_t>(ks) * rt * (BN / ks + 4) * 4;
        if (smem < need) smem = need;
    }
    e = cudaFuncSetAttribute(gemm_tc_kernel<BN, NMAJ, AF32, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    dim3 grid(mtiles * ks, ntiles, p.G);
    ProjEpi none{};
    return launch_dependent(gemm_tc_kernel<BN, NMAJ, AF32, false>, grid, dim3(kGemmThreads), smem, st, ks, q, ma, mb,
                            mb, mb, rope ? *rope : none);
}

// The projection: h [M = batch n_new, hidden] against W^DKV (rank rows), W^KR
// (d_rope rows, one column tile) and W^Q (H (d_nope + d_rope) rows, or none).
template <int BN>
cudaError_t launch_proj(const mla_dims &d, const CacheView &c, int batch, int n_new, const void *h,
                        const void *w_dkv, const void *w_kr, const void *w_q, const int32_t *start_pos, void *q_nope,
                        void *q_pe, unsigned *status, cudaStream_t st)
{
    cudaError_t e = get_encoder();
    if (e != cudaSuccess) return e;
    GroupGemm p{};
    p.M = batch * n_new;
    p.K = d.hidden;
    p.G = 1;
    p.hpg = 1;
    p.blk = 1;
    p.A = h;
    p.a_f32 = 0;
    p.lda = d.hidden;
    p.status = status;
    const int nq = w_q ? d.num_heads * (d.d_nope + d.d_rope) : 0;
    const int rope_rows = d.d_rope < BN ? d.d_rope : BN, q_rows = nq < BN ? nq : BN;
    ProjEpi pe{};
    pe.cache = c;
    pe.start_pos = start_pos;
    pe.q_nope = static_cast<uint16_t *>(q_nope);
    pe.q_pe = static_cast<uint16_t *>(q_pe);
    pe.n_new = n_new;
    pe.rank = d.rank;
    pe.d_rope = d.d_rope;
    pe.d_nope = d.d_nope;
    pe.heads = d.num_heads;
    pe.style = d.rope_style;
    pe.turns = rope_turns(d.d_rope, d.rope_base);
    pe.tiles_lat = d.rank / BN;
    pe.box_bytes[0] = BN * 128;
    pe.box_bytes[1] = static_cast<uint32_t>(rope_rows) * 128;
    pe.box_bytes[2] = static_cast<uint32_t>(q_rows) * 128;
    const int rblk = rows_per_tile(p);
    CUtensorMap ma, m0, m1, m2;
    if (!encode_a(p, rblk, false, &ma) || !encode_kmajor(w_dkv, d.rank, d.hidden, BN, &m0) ||
        !encode_kmajor(w_kr, d.d_rope, d.hidden, rope_rows, &m1))
        return cudaErrorInvalidValue;
    if (w_q) {
        if (!encode_kmajor(w_q, nq, d.hidden, q_rows, &m2)) return cudaErrorInvalidValue;
    } else {
        m2 = m0;  // never read: no query tiles
    }
    const int tiles = pe.tiles_lat + 1 + (nq + BN - 1) / BN;
    p.N = tiles * BN;
    size_t smem = 0;
    p.stages = ring_stages<BN, false>(p.K, &smem);
    p.rblk = rblk;
    p.ksplit = 1;
    e = cudaFuncSetAttribute(gemm_tc_kernel<BN, false, false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    dim3 grid((p.M + rblk - 1) / rblk, tiles, 1);
    return launch_dependent(gemm_tc_kernel<BN, false, false, true>, grid, dim3(kGemmThreads), smem, st, 1, p, ma, m0,
                            m1, m2, pe);
}

}  // namespace

// The absorption GEMM with the positional-query rotation in its epilogue
// warps (N-major W_UK, bf16 q_nope).
cudaError_t launch_absorb_gemm(const GroupGemm &p, const mla_dims &d, const void *q_pe, const int32_t *kv_len,
                               int q_len, cudaStream_t st)
{
    if (p.M <= 0 || p.N <= 0 || p.G <= 0) return cudaSuccess;
    ProjEpi r{};
    r.rope_src = static_cast<const uint16_t *>(q_pe);
    r.kv_len = kv_len;
    r.q_len = q_len;
    r.heads = d.num_heads;
    r.rank = d.rank;
    r.d_rope = d.d_rope;
    r.style = d.rope_style;
    r.turns = rope_turns(d.d_rope, d.rope_base);
    const bool narrow = p.N <= 64 || p.M <= 32;
    return narrow ? launch_tc<64, true, false>(p, st, &r) : launch_tc<128, true, false>(p, st, &r);
}

cudaError_t launch_group_gemm(const GroupGemm &p, cudaStream_t st)
{
    if (p.M <= 0 || p.N <= 0 || p.G <= 0) return cudaSuccess;
    // column tile: 64 for narrow outputs and for few rows (more CTAs stream the
    // weight), else 128
    const bool narrow = p.N <= 64 || p.M <= 32;
    if (p.a_f32) {
        if (p.b_nmajor) return narrow ? launch_tc<64, true, true>(p, st) : launch_tc<128, true, true>(p, st);
        return narrow ? launch_tc<64, false, true>(p, st) : launch_tc<128, false, true>(p, st);
    }
    if (p.b_nmajor) return narrow ? launch_tc<64, true, false>(p, st) : launch_tc<128, true, false>(p, st);
    return narrow ? launch_tc<64, false, false>(p, st) : launch_tc<128, false, false>(p, st);
}

cudaError_t launch_project(const mla_dims &d, const CacheView &c, int batch, int n_new, const void *h,
                           const void *w_dkv, const void *w_kr, const void *w_q, const int32_t *start_pos,
                           void *q_nope, void *q_pe, unsigned *status, cudaStream_t st)
{
    if (batch <= 0 || n_new <= 0) return cudaSuccess;
    // 128-column tiles once there are enough rows to be tensor-bound and the
    // latent splits into whole 128-column tiles; 64 otherwise.  256-column
    // tiles when they take fewer waves of CTAs by more than their extra bytes
    // per K chunk (A 16 KB + B 32 KB against 16 + 16): the row tiles times the
    // column tiles just past one wave at 128 (640 rows: 185 CTAs -> 95).
    const int rows = batch * n_new;
    if (rows > 32 && d.rank % 128 == 0) {
        if (d.rank % 256 == 0) {
            int dev = 0, sms = 0;
            cudaGetDevice(&dev);
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            const int nq = w_q ? d.num_heads * (d.d_nope + d.d_rope) : 0;
            const int64_t mt = (rows + 127) / 128;
            auto waves = [&](int bn) { return (mt * (d.rank / bn + 1 + (nq + bn - 1) / bn) + sms - 1) / sms; };
            if (sms > 0 && waves(256) * 48 < waves(128) * 32)
                return launch_proj<256>(d, c, batch, n_new, h, w_dkv, w_kr, w_q, start_pos, q_nope, q_pe, status, st);
        }
        return launch_proj<128>(d, c, batch, n_new, h, w_dkv, w_kr, w_q, start_pos, q_nope, q_pe, status, st);
    }
    return launch_proj<64>(d, c, batch, n_new, h, w_dkv, w_kr, w_q, start_pos, q_nope, q_pe, status, st);
}

}  // namespace gbmla
