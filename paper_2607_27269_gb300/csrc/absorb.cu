// mla_absorb_q: latent query q_lat = W_UK[g]^T q_nope (attention "through
// absorbed projections", Sec. 1; Eq. 5 read right to left) and the positional
// query rotated to its own position (Sec. 3.1).
//
// A persistent tensor-core kernel, one CTA per SM: the work is a list of items
// (KV group g, tile of up to 128 query rows of the group, slice of 64, 128 or
// 256 latent columns), and each CTA walks its share of the list with the loads
// of the next item, the MMAs of this one and the epilogue of the previous one
// in flight at once (a TMA ring of K chunks, two TMEM accumulators, the output
// staged in shared memory and written by TMA stores).  A CTA per item would pay
// its prologue, first load and epilogue in sequence, with the item count just
// past one wave of CTAs (paged batch of 128 x 5 queries x 32 heads: 640 GEMM
// tiles over 608 CTA slots).  Shapes it does not serve, and few rows against a
// deep K, go to the grouped GEMM of gemm.cu.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace gbmla {
namespace {

constexpr int kAbThreads = 256;   // warp 0 TMA, warp 1 MMA, warps 2-3 positional queries, warps 4-7 epilogue
constexpr int kAbEpiThreads = 128;
constexpr int kAbStages = 3;      // K-chunk stages of (A 16 KB, B up to 32 KB)
constexpr int kAbMaxN = 256;      // most latent columns per item (one TMEM accumulator)

struct AbArgs {
    int M;          // rows per group: batch * q_len * hpg
    int G, hpg, H;  // groups, heads per group, heads
    int K;          // d_nope (a multiple of 64, <= 256)
    int rank, ni;   // latent width, columns per item (ni | rank, ni <= 256, a multiple of 64)
    int R, RT;      // row blocks (of hpg rows) per tile, rows per tile
    int mt, nh;     // row tiles per group, column slices per row tile
    int items;
    int ldc;        // q_abs row length: rank + d_rope
    int q_len, d_rope, style;
    RopeTurns turns;
    const uint16_t *q_pe;
    const int32_t *kv_len;
    uint16_t *q_abs;
    unsigned *status;
};

struct __align__(8) AbBars {
    uint64_t full[kAbStages], empty[kAbStages];
    uint64_t tfull[2], tempty[2];
    uint64_t drain;
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

__device__ __forceinline__ void unpack8(const uint4 v, float *x)
{
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        x[2 * e] = __uint_as_float(w[e] << 16);
        x[2 * e + 1] = __uint_as_float(w[e] & 0xFFFF0000u);
    }
}

__device__ __forceinline__ uint4 pack8(const float *y)
{
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const __nv_bfloat162 b = __floats2bfloat162_rn(y[2 * e], y[2 * e + 1]);
        w[e] = *reinterpret_cast<const uint32_t *>(&b);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// eight fp32 bit patterns -> eight bf16 (round to nearest even)
__device__ __forceinline__ uint4 pack8u(const uint32_t *v)
{
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const __nv_bfloat162 b = __floats2bfloat162_rn(__uint_as_float(v[2 * e]), __uint_as_float(v[2 * e + 1]));
        w[e] = *reinterpret_cast<const uint32_t *>(&b);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

__device__ __forceinline__ void tma_store_5d(const CUtensorMap *map, uint32_t src, int32_t c0, int32_t c1, int32_t c2,
                                             int32_t c3, int32_t c4)
{
    asm volatile("cp.async.bulk.tensor.5d.global.shared::cta.bulk_group [%0, {%1, %2, %3, %4, %5}], [%6];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(c4), "r"(src)
                 : "memory");
}

__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// every committed store has finished reading shared memory / has completed
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait0() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void named_bar_sync(int id, int threads)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

__global__ void __launch_bounds__(kAbThreads) absorb_kernel(const __grid_constant__ AbArgs a,
                                                            const __grid_constant__ CUtensorMap map_a,
                                                            const __grid_constant__ CUtensorMap map_b,
                                                            const __grid_constant__ CUtensorMap map_c)
{
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ AbBars bars;
    __shared__ uint32_t tmem_base;
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~static_cast<uintptr_t>(1023));
    constexpr int kABytes = 128 * 128;            // 128 rows x 64 K, SW128 K-major
    const uint32_t b_bytes = static_cast<uint32_t>(a.ni) * 128;  // 64 K rows x ni columns, SW128 N-major (64-column blocks)
    unsigned char *sa = smem;                      // kAbStages x A chunk
    unsigned char *sb = sa + kAbStages * kABytes;  // kAbStages x B chunk
    unsigned char *stage = sb + kAbStages * (kAbMaxN * 128);  // output staging: ni / 64 blocks of RT rows x 128 B
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nkc = a.K / 64;
    const uint64_t lim = kWaitLimitNs;

    if (tid == 0) {
        for (int s = 0; s < kAbStages; ++s) {
            mbar_init(&bars.full[s], 1);
            mbar_init(&bars.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars.tfull[b], 1);
            mbar_init(&bars.tempty[b], kAbEpiThreads / 32);
        }
        mbar_init(&bars.drain, 1);
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(smem_u32(&tmem_base), 2 * a.ni);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    // the queries come from the previous launch; this kernel writes no cache,
    // so its dependents (the attention core) may launch at once
    griddep_wait();
    griddep_launch_dependents();
    const uint32_t tmem = tmem_base;
    const int nmine = a.items > static_cast<int>(blockIdx.x)
                          ? (a.items - 1 - static_cast<int>(blockIdx.x)) / static_cast<int>(gridDim.x) + 1
                          : 0;
    auto item_of = [&](int j, int *g, int *mt, int *nh) {
        const int it = static_cast<int>(blockIdx.x) + j * static_cast<int>(gridDim.x);
        *nh = it % a.nh;
        const int gm = it / a.nh;
        *mt = gm % a.mt;
        *g = gm / a.mt;
    };

    if (warp == 0) {
        // ---- K chunks of A (query rows) and B (W_UK columns) by TMA, item after item
        if (lane == 0) {
            tc::prefetch_tensormap(&map_a);
            tc::prefetch_tensormap(&map_b);
            tc::prefetch_tensormap(&map_c);
        }
        int issued = 0;
        for (int job = 0; job < nmine * nkc; ++job) {
            const int j = job / nkc, kc = job - j * nkc, s = job % kAbStages, round = job / kAbStages;
            if (round >= 1 && !__all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.empty[s]), (round - 1) & 1, lim))) {
                if (lane == 0) record_status(a.status, kStatusTimeout);
                break;
            }
            issued = job + 1;
            // lane 0 loads the A box, lane 1 the B box (one tensor-TMA
            // instruction occupies its thread for a long time, whatever its size)
            int g, mt, nh;
            item_of(j, &g, &mt, &nh);
            const uint32_t fb = smem_u32(&bars.full[s]);
            if (lane == 0) tc::mbar_arrive_expect_tx(fb, static_cast<uint32_t>(a.RT) * 128 + b_bytes);
            __syncwarp();
            if (lane == 0) tma_load_4d(smem_u32(sa + s * kABytes), &map_a, 64 * kc, 0, g, mt * a.R, fb);
            if (lane == 1)
                tc::tma_load_3d(smem_u32(sb + s * (kAbMaxN * 128)), &map_b, 0, g * a.K + 64 * kc, nh * (a.ni / 64),
                                fb);
            __syncwarp();
        }
        // no copy may still be landing when the CTA exits: wait (bounded) for
        // the last load of every stage; after a normal run all have landed
        for (int job = issued > kAbStages ? issued - kAbStages : 0; job < issued; ++job)
            if (!__all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.full[job % kAbStages]), (job / kAbStages) & 1, lim)))
                if (lane == 0) record_status(a.status, kStatusTimeout);
    } else if (warp == 1) {
        // ---- MMAs: item j accumulates in TMEM buffer j % 2 (converged warp, one elected lane issues)
        const uint32_t idesc = tc::idesc_bf16_f32(128, a.ni, false, true);
        const uint64_t da = tc::smem_desc(0, 16, 1024, tc::kSwizzle128B);
        const uint64_t db = tc::smem_desc(0, 64 * 128, 1024, tc::kSwizzle128B);
        auto with_addr = [](uint64_t tmpl, uint32_t saddr) {
            return tmpl | static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
        };
        bool ok = true;
        for (int j = 0; j < nmine && ok; ++j) {
            const int buf = j & 1;
            if (j >= 2) ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.tempty[buf]), ((j >> 1) - 1) & 1, lim));
            if (!ok) break;
            tc::fence_after_sync();
            const uint32_t d = tmem + static_cast<uint32_t>(buf * a.ni);
            for (int kc = 0; kc < nkc && ok; ++kc) {
                const int job = j * nkc + kc, s = job % kAbStages;
                ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.full[s]), (job / kAbStages) & 1, lim));
                if (!ok) break;
                tc::fence_after_sync();
                const uint32_t ab = smem_u32(sa + s * kABytes), bb = smem_u32(sb + s * (kAbMaxN * 128));
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    tc::mma_bf16_elect(d, with_addr(da, ab + kk * 32), with_addr(db, bb + kk * 16 * 128), idesc,
                                       (kc | kk) != 0);
                tc::commit_elect(smem_u32(&bars.empty[s]));
            }
            if (ok) tc::commit_elect(smem_u32(&bars.tfull[buf]));
        }
        if (!ok && lane == 0) record_status(a.status, kStatusTimeout);
        tc::commit_elect(smem_u32(&bars.drain));
        if (!__all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.drain), 0, lim)) && lane == 0)
            record_status(a.status, kStatusTimeout);
    } else if (warp < 4) {
        // ---- positional queries.  The tokens of a row tile are split over
        // its column slices, so that every item carries a share.  A unit of
        // work is (token, eight pairs): eight angles, applied to those pairs
        // of every head of the group, which sit in two 16-byte chunks of the
        // row (k .. k + 7 and half + k .. half + k + 7 in the half-split
        // style, 2k .. 2k + 15 interleaved).
        const int half = a.d_rope / 2, n8 = half / 8;
        for (int j = 0; j < nmine; ++j) {
            int g, mt, nh;
            item_of(j, &g, &mt, &nh);
            const int m0 = mt * a.RT;
            const int ntok = min(a.RT, a.M - m0) / a.hpg, tok0 = m0 / a.hpg;
            const int t_lo = ntok * nh / a.nh, t_hi = ntok * (nh + 1) / a.nh;
            for (int it = tid - 64; it < (t_hi - t_lo) * n8; it += 64) {
                const int kg = it % n8, bi = tok0 + t_lo + it / n8;  // bi = b q_len + i
                const int b = bi / a.q_len, i = bi - b * a.q_len;
                const int64_t pos = static_cast<int64_t>(__ldg(a.kv_len + b)) - a.q_len + i;
                const int e0 = a.style == 0 ? 8 * kg : 16 * kg, e1 = a.style == 0 ? half + 8 * kg : 16 * kg + 8;
                const int64_t row0 = static_cast<int64_t>(bi) * a.H + static_cast<int64_t>(g) * a.hpg;
                float cs[8], sn[8];
                for (int h0 = 0; h0 < a.hpg; h0 += 4) {
                    uint4 va[4], vb[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        if (h0 + u < a.hpg) {
                            const uint16_t *src = a.q_pe + (row0 + h0 + u) * a.d_rope;
                            va[u] = __ldg(reinterpret_cast<const uint4 *>(src + e0));
                            vb[u] = __ldg(reinterpret_cast<const uint4 *>(src + e1));
                        }
                    if (h0 == 0) {
#pragma unroll
                        for (int q = 0; q < 8; ++q) rope_cos_sin(pos, a.turns.f[8 * kg + q], &cs[q], &sn[q]);
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        if (h0 + u < a.hpg) {
                            float x[16];
                            unpack8(va[u], x);
                            unpack8(vb[u], x + 8);
                            float y[16];
                            if (a.style == 0) {
#pragma unroll
                                for (int q = 0; q < 8; ++q) {
                                    y[q] = x[q] * cs[q] - x[q + 8] * sn[q];
                                    y[q + 8] = x[q + 8] * cs[q] + x[q] * sn[q];
                                }
                            } else {
#pragma unroll
                                for (int q = 0; q < 8; ++q) {
                                    y[2 * q] = x[2 * q] * cs[q] - x[2 * q + 1] * sn[q];
                                    y[2 * q + 1] = x[2 * q + 1] * cs[q] + x[2 * q] * sn[q];
                                }
                            }
                            uint16_t *dst = a.q_abs + (row0 + h0 + u) * a.ldc + a.rank;
                            *reinterpret_cast<uint4 *>(dst + e0) = pack8(y);
                            *reinterpret_cast<uint4 *>(dst + e1) = pack8(y + 8);
                        }
                }
            }
        }
    } else {
        // ---- epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31 (the tile's
        // rows), converts them to bf16 and stages them in shared memory as
        // the box of one TMA store: 64-column blocks of RT rows of 128 bytes,
        // in the 128-byte swizzle.  Every warp passes the same named barriers
        // for every item: a warp whose wait ran out skips its work from then
        // on but keeps to the barriers.
        const int q = warp & 3, i = q * 32 + lane;
        const bool issuer = warp == 4 && lane == 0;
        const uint32_t t_lane = tmem + (static_cast<uint32_t>(q * 32) << 16);
        const int nblk = a.ni / 64;
        bool ok = true;
        for (int j = 0; j < nmine; ++j) {
            const int buf = j & 1;
            if (ok && !__all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.tfull[buf]), (j >> 1) & 1, lim))) {
                if (lane == 0) record_status(a.status, kStatusTimeout);
                ok = false;
            }
            tc::fence_after_sync();
            int g, mt, nh;
            item_of(j, &g, &mt, &nh);
            if (issuer) bulk_wait_read0();  // the previous item's store has left the staging buffer
            named_bar_sync(1, kAbEpiThreads);
            const uint32_t t_buf = t_lane + static_cast<uint32_t>(buf * a.ni);
#pragma unroll 1
            for (int c = 0; c < nblk && ok; ++c) {
                uint32_t v[4][16];
#pragma unroll
                for (int u = 0; u < 4; ++u) tc::ld_32x32b_x16(t_buf + 64 * c + 16 * u, v[u]);
                tc::wait_ld();
                if (i < a.RT) {
                    // row r of the box (r = c RT + i): 16-byte chunk k at chunk k ^ (r % 8)
                    const int r = c * a.RT + i;
                    unsigned char *row = stage + r * 128;
#pragma unroll
                    for (int k = 0; k < 8; ++k)
                        *reinterpret_cast<uint4 *>(row + ((k ^ (r & 7)) << 4)) = pack8u(&v[k >> 1][8 * (k & 1)]);
                }
            }
            // the accumulator may be overwritten once every warp's loads are done
            tc::fence_before_sync();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(smem_u32(&bars.tempty[buf]));
            tc::fence_proxy_async_smem();
            named_bar_sync(1, kAbEpiThreads);
            if (issuer && ok) {
                tma_store_5d(&map_c, smem_u32(stage), 0, 0, g, mt * a.R, nh * nblk);
                bulk_commit();
            }
        }
        if (issuer) bulk_wait0();
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, 2 * a.ni);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode_ab = nullptr;

cudaError_t get_encoder_ab()
{
    if (g_encode_ab) return cudaSuccess;
    cudaDriverEntryPointQueryResult qr;
    void *fn = nullptr;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &qr);
    if (e != cudaSuccess || qr != cudaDriverEntryPointSuccess || !fn) return e != cudaSuccess ? e : cudaErrorUnknown;
    g_encode_ab = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return cudaSuccess;
}

// The persistent kernel, or cudaErrorNotSupported for a shape it does not serve.
cudaError_t launch_absorb_persistent(const mla_dims &d, int batch, int q_len, const void *q_nope, const void *q_pe,
                                     const int32_t *kv_len, const void *w_uk, void *q_abs, unsigned *status,
                                     cudaStream_t st)
{
    const int H = d.num_heads, G = d.num_kv_groups, hpg = H / G;
    if (d.d_nope % 64 || d.d_nope > 256 || d.rank % 64 || hpg > 128 || d.d_rope > 128 || d.d_rope % 16)
        return cudaErrorNotSupported;
    // 16-byte accesses to the positional parts
    if (reinterpret_cast<uintptr_t>(q_pe) % 16 || reinterpret_cast<uintptr_t>(q_abs) % 16)
        return cudaErrorNotSupported;
    AbArgs a{};
    a.M = batch * q_len * hpg;
    if (a.M <= 0) return cudaSuccess;
    a.G = G;
    a.hpg = hpg;
    a.H = H;
    a.K = d.d_nope;
    a.rank = d.rank;
    // row tiles of whole tokens (hpg rows each), no more tokens than there are
    a.R = 128 / hpg < batch * q_len ? 128 / hpg : batch * q_len;
    a.RT = a.R * hpg;
    a.mt = (a.M + a.RT - 1) / a.RT;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    // 256-column slices, narrowed (down to 64) while the items would fill
    // fewer than half the SMs: few rows (small batches) then still spread
    // their weight reads and stores over more CTAs
    a.ni = d.rank % 256 == 0 ? 256 : d.rank % 128 == 0 ? 128 : 64;
    while (a.ni > 64 && static_cast<int64_t>(G) * a.mt * (d.rank / a.ni) < sms / 2) a.ni /= 2;
    a.nh = d.rank / a.ni;
    a.items = G * a.mt * a.nh;
    const int path = tuning().absorb_path;
    if (path == 2) return cudaErrorNotSupported;
    // Few rows against a deep K (two or more chunks, under a quarter wave of
    // 256-column items): the grouped GEMM.  Both take the same time alone,
    // but in the step, where the attention core starts streaming the cache
    // on the SMs this launch leaves free, the GEMM came out ~1.5 us ahead
    // (8 sequences x 24 heads, d_nope 128).
    const int64_t items256 = static_cast<int64_t>(G) * a.mt * (d.rank >= 256 ? d.rank / 256 : 1);
    if (path == 0 && d.d_nope > 64 && items256 < sms / 4) return cudaErrorNotSupported;
    a.ldc = d.rank + d.d_rope;
    a.q_len = q_len;
    a.d_rope = d.d_rope;
    a.style = d.rope_style;
    a.turns = rope_turns(d.d_rope, d.rope_base);
    a.q_pe = static_cast<const uint16_t *>(q_pe);
    a.kv_len = kv_len;
    a.q_abs = static_cast<uint16_t *>(q_abs);
    a.status = status;
    cudaError_t e = get_encoder_ab();
    if (e != cudaSuccess) return e;
    CUtensorMap ma, mb, mc;
    {
        // A: q_nope rows (K, head in group, group, token), box 64 x hpg x 1 x R
        cuuint64_t dims[4] = {static_cast<cuuint64_t>(d.d_nope), static_cast<cuuint64_t>(hpg),
                              static_cast<cuuint64_t>(G), static_cast<cuuint64_t>(batch) * q_len};
        cuuint64_t strides[3] = {static_cast<cuuint64_t>(d.d_nope) * 2, static_cast<cuuint64_t>(hpg) * d.d_nope * 2,
                                 static_cast<cuuint64_t>(H) * d.d_nope * 2};
        cuuint32_t box[4] = {64u, static_cast<cuuint32_t>(hpg), 1u, static_cast<cuuint32_t>(a.R)};
        cuuint32_t es[4] = {1, 1, 1, 1};
        if (g_encode_ab(&ma, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(q_nope), dims, strides, box, es,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    {
        // B: W_UK [G d_nope rows][rank columns] (N-major) as (column in block,
        // row, 64-column block); box 64 x 64 x ni / 64: the 64-column blocks of
        // one K chunk land one after another (8 KB each), as the MMA reads them
        cuuint64_t dims[3] = {64u, static_cast<cuuint64_t>(G) * d.d_nope, static_cast<cuuint64_t>(d.rank / 64)};
        cuuint64_t strides[2] = {static_cast<cuuint64_t>(d.rank) * 2, 128u};
        cuuint32_t box[3] = {64u, 64u, static_cast<cuuint32_t>(a.ni / 64)}, es[3] = {1, 1, 1};
        if (g_encode_ab(&mb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(w_uk), dims, strides, box, es,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    {
        // C: the latent columns of q_abs as (column in block, head in group,
        // group, token, 64-column block), rows of ldc elements; box 64 x hpg x
        // 1 x R x ni / 64, stored from the staging buffer in one instruction
        cuuint64_t dims[5] = {64u, static_cast<cuuint64_t>(hpg), static_cast<cuuint64_t>(G),
                              static_cast<cuuint64_t>(batch) * q_len, static_cast<cuuint64_t>(d.rank / 64)};
        cuuint64_t strides[4] = {static_cast<cuuint64_t>(a.ldc) * 2, static_cast<cuuint64_t>(hpg) * a.ldc * 2,
                                 static_cast<cuuint64_t>(H) * a.ldc * 2, 128u};
        cuuint32_t box[5] = {64u, static_cast<cuuint32_t>(hpg), 1u, static_cast<cuuint32_t>(a.R),
                             static_cast<cuuint32_t>(a.ni / 64)};
        cuuint32_t es[5] = {1, 1, 1, 1, 1};
        if (g_encode_ab(&mc, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, q_abs, dims, strides, box, es,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    }
    // ring stages (A 16 KB + B 32 KB each) and the output staging (ni / 64 blocks of 16 KB)
    const size_t smem = 1024 + static_cast<size_t>(kAbStages) * (128 * 128 + kAbMaxN * 128) +
                        static_cast<size_t>(a.ni / 64) * (128 * 128);
    if ((e = cudaFuncSetAttribute(absorb_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(smem))) != cudaSuccess)
        return e;
    const int grid = a.items < sms ? a.items : sms;
    return launch_dependent(absorb_kernel, dim3(grid), dim3(kAbThreads), smem, st, 1, a, ma, mb, mc);
}

}  // namespace

cudaError_t launch_absorb(const mla_dims &d, int batch, int q_len, const void *q_nope, const void *q_pe,
                          const int32_t *kv_len, const void *w_uk, void *q_abs, unsigned *status,
                          cudaStream_t st)
{
    const cudaError_t pe = launch_absorb_persistent(d, batch, q_len, q_nope, q_pe, kv_len, w_uk, q_abs, status, st);
    if (pe != cudaErrorNotSupported) return pe;  // else the grouped GEMM serves the shape
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
