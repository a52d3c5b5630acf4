// mla_gqa_*: decode attention of the original GQA draft (Sec. 3.1, Eqs. 1-4),
// the model the converted MLA draft replaces, at the same shapes, so that the
// two caches can be compared byte for byte and second for second.  Each KV
// group g of sequence b keeps its own key cache K (stored rotated to its
// position) and value cache V; unit u = b * G + g is one such (sequence,
// group), with kv_len[b] tokens.
//
// One CTA = one split-KV partition of the units' 128-token tiles (the same
// partition as the MLA path, over units instead of sequences), 256 threads:
//   warp 0      TMA producer: the K tile of every tile into the K ring, the V
//               tile into the V ring (each read once from HBM);
//   warp 1      MMA issuer: S[rows, 128 tok] = Q K^T into one of two TMEM
//               buffers, O[rows, d] += P V into TMEM;
//   warps 4..7  one thread per query row (row r = position i * hpg + head hh
//               of the group): stages the rotated queries of each unit,
//               runs the online softmax of its row (lazy rescaling), writes
//               its row of P, and at the end of a unit writes its partial.
// The rows of a unit (q_len * hpg <= 128) fill the MMA's M = 128; rows past
// them are padding.  Every wait is bounded; a timeout is recorded in the
// status word and the CTA winds down.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace gbmla {
namespace {

constexpr int kGqaThreads = 256;
constexpr int kTokTile = MLA_SPLIT_TILE;  // 128 tokens per tile
constexpr int kSmBase = 128;              // first softmax thread (warp 4)
constexpr int kMaxRing = 8;

struct GqaArgs {
    int batch, q_len, groups, hpg, rows, max_kv, num_splits;
    int paged, bt_stride, num_pages, nk, nv;  // nk / nv: K / V ring slots
    float scale_log2;
    int style;
    const int32_t *kv_len;
    const int32_t *block_table;
    const uint16_t *q;  // [B, q_len, H, DK]
    float *o_part, *lse_part;
    unsigned *status;
    RopeTurns turns;
};

struct __align__(8) GqaBars {
    uint64_t k_full[kMaxRing], k_empty[kMaxRing], v_full[kMaxRing], v_empty[kMaxRing];
    uint64_t s_full[2], s_free[2], p_full, pv_done, q_full;
};

// Units [u0, ..) and their tiles, walked in the partition's order.
struct UnitWalk {
    const int32_t *kv;
    int groups, q_len, max_kv, batch;
    int u;             // current unit
    int64_t start, nb; // first flat tile of the unit, its tile count
    int64_t t, t_end;
    __device__ void init(const int32_t *kv_len, int groups_, int q_len_, int max_kv_, int units, int64_t tb,
                         int64_t te)
    {
        kv = kv_len;
        groups = groups_;
        q_len = q_len_;
        max_kv = max_kv_;
        batch = units;
        t = tb;
        t_end = te;
        start = 0;
        nb = 0;
        for (u = 0; u < units; ++u) {
            nb = seq_tiles(kv[u / groups], q_len, max_kv);
            if (start + nb > t) break;
            start += nb;
        }
    }
    __device__ int tile() const { return static_cast<int>(t - start); }
    __device__ bool first(int64_t tb) const { return t == tb || t == start; }
    __device__ bool last() const { return t + 1 == t_end || t + 1 == start + nb; }
    __device__ void next()
    {
        ++t;
        if (t < t_end && t >= start + nb) {
            start += nb;
            for (++u; u < batch; ++u) {
                nb = seq_tiles(kv[u / groups], q_len, max_kv);
                if (nb > 0) break;
            }
        }
    }
};

__device__ __forceinline__ bool wait_all(uint64_t *bar, uint32_t parity)
{
    return __all_sync(0xffffffffu, mbar_wait(smem_u32(bar), parity, kWaitLimitNs));
}

// byte offset of 16-byte chunk j of row r in a 128-row SW128 K-major atom
__device__ __forceinline__ uint32_t sw128(int r, int j)
{
    return static_cast<uint32_t>((r >> 3) * 1024 + (r & 7) * 128 + ((j ^ (r & 7)) << 4));
}

__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Query row r of the unit, rotated to position pos (RoPE over the whole head,
// fp32), into the SW128 K-major Q tile; a null src writes a zero row (padding).
template <int D>
__device__ __forceinline__ void stage_query(unsigned char *q_buf, int r, const uint16_t *src, int64_t pos, int style,
                                            const RopeTurns &turns)
{
    float x[D];
    if (src) {
#pragma unroll
        for (int v = 0; v < D / 8; ++v) {
            const uint4 raw = reinterpret_cast<const uint4 *>(src)[v];
            const uint32_t wd[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                x[8 * v + 2 * e] = __uint_as_float(wd[e] << 16);
                x[8 * v + 2 * e + 1] = __uint_as_float(wd[e] & 0xffff0000u);
            }
        }
        if (style == 0) {
#pragma unroll
            for (int k = 0; k < D / 2; ++k) {
                float cs, sn;
                rope_cos_sin(pos, turns.f[k], &cs, &sn);
                const float a0 = x[k], a1 = x[k + D / 2];
                x[k] = a0 * cs - a1 * sn;
                x[k + D / 2] = a1 * cs + a0 * sn;
            }
        } else {
#pragma unroll
            for (int k = 0; k < D / 2; ++k) {
                float cs, sn;
                rope_cos_sin(pos, turns.f[k], &cs, &sn);
                const float a0 = x[2 * k], a1 = x[2 * k + 1];
                x[2 * k] = a0 * cs - a1 * sn;
                x[2 * k + 1] = a1 * cs + a0 * sn;
            }
        }
    } else {
#pragma unroll
        for (int e = 0; e < D; ++e) x[e] = 0.f;
    }
#pragma unroll
    for (int at = 0; at < D / 64; ++at)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            uint32_t wd[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const __nv_bfloat162 h2 = __floats2bfloat162_rn(x[64 * at + 8 * j + 2 * e], x[64 * at + 8 * j + 2 * e + 1]);
                wd[e] = *reinterpret_cast<const uint32_t *>(&h2);
            }
            *reinterpret_cast<uint4 *>(q_buf + at * 128 * 128 + sw128(r, j)) = make_uint4(wd[0], wd[1], wd[2], wd[3]);
        }
}

template <int D>
__global__ void __launch_bounds__(kGqaThreads) gqa_attn_kernel(const __grid_constant__ GqaArgs a,
                                                              const __grid_constant__ CUtensorMap map_k,
                                                              const __grid_constant__ CUtensorMap map_v)
{
    constexpr int KA = D / 64;                  // 64-column atoms of a K or V tile
    constexpr uint32_t kTileBytes = kTokTile * D * 2;
    constexpr uint32_t kAtom = 128 * 128;       // 128 rows x 64 columns bf16
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ GqaBars bars;
    __shared__ uint32_t tmem_base;
    __shared__ int64_t red64[64];
    __shared__ int abort_flag;
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~static_cast<uintptr_t>(1023));
    unsigned char *q_buf = smem;                       // KA atoms: Q [128 rows, D]
    unsigned char *p_buf = q_buf + KA * kAtom;         // 2 atoms: P [128 rows, 128 tokens]
    unsigned char *k_ring = p_buf + 2 * kAtom;         // nk tiles
    unsigned char *v_ring = k_ring + a.nk * kTileBytes; // nv tiles
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int part = blockIdx.y;
    const int units = a.batch * a.groups;
    const int nw = (a.rows + 31) / 32;  // softmax warps holding real rows

    if (tid == 0) {
        for (int s = 0; s < kMaxRing; ++s) {
            mbar_init(&bars.k_full[s], 1);
            mbar_init(&bars.k_empty[s], 1);
            mbar_init(&bars.v_full[s], 1);
            mbar_init(&bars.v_empty[s], 1);
        }
        for (int j = 0; j < 2; ++j) {
            mbar_init(&bars.s_full[j], 1);
            mbar_init(&bars.s_free[j], nw);
        }
        mbar_init(&bars.p_full, nw);
        mbar_init(&bars.pv_done, 1);
        mbar_init(&bars.q_full, nw);
        abort_flag = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(smem_u32(&tmem_base), 512);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    // the cache is final when this kernel runs (a cache writer releases its
    // dependents only on completion); the queries come from the previous
    // launch: the softmax warps wait before they read them
    griddep_launch_dependents();
    const int64_t T = block_tile_sum(a.kv_len, units, a.q_len, a.max_kv, red64, a.groups);
    const int64_t t_begin = T ? part_begin(part, T, a.num_splits) : 0;
    const int64_t t_end = T ? part_begin(part + 1, T, a.num_splits) : 0;
    const int n_items = static_cast<int>(t_end - t_begin);
    const uint32_t tmem = tmem_base;
    auto fail = [&]() {
        record_status(a.status, kStatusTimeout);
        abort_flag = 1;
    };

    if (warp == 0 && n_items > 0) {
        // ================================================================ TMA producer
        if (lane == 0) {
            tc::prefetch_tensormap(&map_k);
            tc::prefetch_tensormap(&map_v);
        }
        UnitWalk w;
        w.init(a.kv_len, a.groups, a.q_len, a.max_kv, units, t_begin, t_end);
        for (int it = 0; it < n_items; ++it, w.next()) {
            // where the tile lives: one 128-row box (contiguous) or a 64-row box per page
            const int u = w.u, j = w.tile();
            int nh = 1;
            int32_t blk[2] = {u, 0}, tok0[2] = {j * kTokTile, 0};
            if (a.paged) {
                const int kv = a.kv_len[u / a.groups];
                nh = kv - j * kTokTile > 64 ? 2 : 1;
                for (int h = 0; h < nh; ++h) {
                    const int32_t pg = a.block_table[static_cast<int64_t>(u) * a.bt_stride + 2 * j + h];
                    if (pg < 0 || pg >= a.num_pages) {
                        if (lane == 0) record_status(a.status, kStatusBounds);
                        nh = h;
                        break;
                    }
                    blk[h] = pg;
                    tok0[h] = 0;
                }
            }
            const uint32_t bytes = static_cast<uint32_t>(nh) * (a.paged ? 64u : 128u) * D * 2;
            for (int kind = 0; kind < 2; ++kind) {  // K, then V
                const int ring = kind == 0 ? a.nk : a.nv;
                const int s = it % ring, round = it / ring;
                uint64_t *empty = kind == 0 ? &bars.k_empty[s] : &bars.v_empty[s];
                uint64_t *full = kind == 0 ? &bars.k_full[s] : &bars.v_full[s];
                if (round > 0 && !wait_all(empty, (round - 1) & 1)) {
                    if (lane == 0) fail();
                    it = n_items;
                    break;
                }
                if (lane == 0) {
                    const uint32_t dst = smem_u32((kind == 0 ? k_ring : v_ring) + s * kTileBytes);
                    const CUtensorMap *map = kind == 0 ? &map_k : &map_v;
                    // (the arrive completes the phase at once when a bad page left nothing to load)
                    tc::mbar_arrive_expect_tx(smem_u32(full), bytes);
                    for (int at = 0; at < KA; ++at)
                        for (int h = 0; h < nh; ++h)
                            tc::tma_load_3d(dst + at * kAtom + h * 64 * 128, map, 64 * at, tok0[h], blk[h],
                                            smem_u32(full));
                }
                __syncwarp();
            }
        }
    } else if (warp == 1 && n_items > 0) {
        // ================================================================ MMA issuer
        const uint32_t idesc_qk = tc::idesc_bf16_f32(128, 128, false, false);
        const uint32_t idesc_pv = tc::idesc_bf16_f32(128, D, false, true);
        const uint64_t d_k = tc::smem_desc(0, 16, 1024, tc::kSwizzle128B);           // K-major operands
        const uint64_t d_v = tc::smem_desc(0, kAtom, 1024, tc::kSwizzle128B);        // V: N-major
        auto with_addr = [](uint64_t tmpl, uint32_t saddr) {
            return tmpl | static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
        };
        const uint32_t q_base = smem_u32(q_buf), p_base = smem_u32(p_buf);
        const uint32_t o_tmem = tmem + 256;  // S buffers at columns [0, 128) and [128, 256)
        UnitWalk w;
        w.init(a.kv_len, a.groups, a.q_len, a.max_kv, units, t_begin, t_end);
        bool ok = true;
        int seq = 0;  // units begun (q_full phases)
        auto qk = [&](int it) {
            const int s = it % a.nk;
            if (it >= 2) ok = ok && wait_all(&bars.s_free[it & 1], ((it - 2) >> 1) & 1);
            ok = ok && wait_all(&bars.k_full[s], (it / a.nk) & 1);
            if (!ok) return;
            tc::fence_after_sync();
            const uint32_t kb = smem_u32(k_ring + s * kTileBytes);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
                const uint32_t off = (kk >> 2) * kAtom + (kk & 3) * 32;
                tc::mma_bf16_elect(tmem + (it & 1) * 128, with_addr(d_k, q_base + off), with_addr(d_k, kb + off),
                                   idesc_qk, kk > 0);
            }
            tc::commit_elect(smem_u32(&bars.k_empty[s]));
            tc::commit_elect(smem_u32(&bars.s_full[it & 1]));
        };
        auto pv = [&](int it, bool first, int u, int j) {
            const int s = it % a.nv;
            ok = ok && wait_all(&bars.p_full, it & 1);
            ok = ok && wait_all(&bars.v_full[s], (it / a.nv) & 1);
            if (!ok) return;
            tc::fence_after_sync();
            // value rows at or past the unit's end (never loaded, or past kv_len)
            // may hold anything; their weights are 0, and 0 x NaN is NaN: zero them
            const int valid = min(a.kv_len[u / a.groups] - j * kTokTile, kTokTile);
            if (valid < kTokTile) {
                unsigned char *vt = v_ring + s * kTileBytes;
                for (int at = 0; at < KA; ++at)
                    for (int rr = valid + lane; rr < kTokTile; rr += 32)
#pragma unroll
                        for (int ch = 0; ch < 8; ++ch)
                            *reinterpret_cast<uint4 *>(vt + at * kAtom + (rr >> 3) * 1024 + (rr & 7) * 128 + ch * 16) =
                                make_uint4(0u, 0u, 0u, 0u);
                tc::fence_proxy_async_smem();
                __syncwarp();
            }
            const uint32_t vb = smem_u32(v_ring + s * kTileBytes);
#pragma unroll
            for (int kk = 0; kk < kTokTile / 16; ++kk) {
                const uint32_t pa = p_base + (kk >> 2) * kAtom + (kk & 3) * 32;
                tc::mma_bf16_elect(o_tmem, with_addr(d_k, pa), with_addr(d_v, vb + kk * 16 * 128), idesc_pv,
                                   !(first && kk == 0));
            }
            tc::commit_elect(smem_u32(&bars.v_empty[s]));
            tc::commit_elect(smem_u32(&bars.pv_done));
        };
        // QK(t + 1) goes ahead of PV(t) within a unit; at a unit boundary PV(t)
        // goes first (the next unit's queries are staged after this unit's end)
        ok = wait_all(&bars.q_full, 0);
        seq = 1;
        if (ok) qk(0);
        for (int it = 0; it < n_items && ok; ++it) {
            const bool first = w.first(t_begin), last = w.last();
            const int u = w.u, j = w.tile();
            if (!last && it + 1 < n_items) qk(it + 1);
            pv(it, first, u, j);
            w.next();
            if (last && it + 1 < n_items && ok) {
                ok = wait_all(&bars.q_full, seq & 1);
                ++seq;
                if (ok) qk(it + 1);
            }
        }
        if (!ok && lane == 0) fail();
    } else if (warp >= 4 && warp < 4 + nw) {
        // ================================================================ softmax / epilogue
        // (only the warps holding real rows: nw = ceil(rows / 32))
        griddep_wait();  // the queries come from the previous launch
        const int r = tid - kSmBase;                 // query row = TMEM lane
        const int qq = warp & 3;                     // lane quarter
        const uint32_t lane_addr = tmem + (static_cast<uint32_t>(qq * 32) << 16);
        const bool row_ok = r < a.rows;
        const int i = r / a.hpg, hh = r % a.hpg;     // query position and head in the group
        UnitWalk w;
        w.init(a.kv_len, a.groups, a.q_len, a.max_kv, units, t_begin, t_end);
        float m_used = -INFINITY, l = 0.f;
        bool ok = true;
        int64_t pos = 0;  // this row's query position in the current unit
        for (int it = 0; it < n_items && ok; ++it, w.next()) {
            const int u = w.u, b = u / a.groups, g = u % a.groups;
            const int kv = a.kv_len[b];
            if (w.first(t_begin)) {
                // ---- stage the unit's rotated queries: row r = (i, hh), head g * hpg + hh
                pos = static_cast<int64_t>(kv) - a.q_len + i;
                const uint16_t *src =
                    a.q + ((static_cast<int64_t>(b) * a.q_len + i) * (a.groups * a.hpg) + g * a.hpg + hh) * D;
                stage_query<D>(q_buf, r, row_ok ? src : nullptr, pos, a.style, a.turns);
                tc::fence_proxy_async_smem();
                __syncwarp();
                tc::mbar_arrive_elect(smem_u32(&bars.q_full));
                m_used = -INFINITY;
                l = 0.f;
            }
            // ---- scores of tile it: pass 1 the row maximum, pass 2 the weights
            ok = wait_all(&bars.s_full[it & 1], (it >> 1) & 1);
            if (!ok) break;
            tc::fence_after_sync();
            const uint32_t s_addr = lane_addr + (it & 1) * 128;
            // causal mask and the tile's tail: token t0 + c is visible iff <= pos and < kv
            const int64_t t0 = static_cast<int64_t>(w.tile()) * kTokTile;
            const int vis = row_ok ? static_cast<int>(min(pos + 1, static_cast<int64_t>(kv)) - t0) : 0;
            float mx = -INFINITY;
#pragma unroll 1
            for (int c = 0; c < kTokTile; c += 16) {
                uint32_t v[16];
                tc::ld_32x32b_x16(s_addr + c, v);
                tc::wait_ld();
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    if (c + e < vis) mx = fmaxf(mx, __uint_as_float(v[e]));
            }
            mx = mx == -INFINITY ? mx : mx * a.scale_log2;
            const bool over = row_ok && mx != -INFINITY && (m_used == -INFINITY || mx > m_used + 8.f);
            float alpha = 1.f;
            if (over) {
                alpha = m_used == -INFINITY ? 0.f : ex2(m_used - mx);
                m_used = mx;
                l *= alpha;
            }
            // P(it) overwrites P(it - 1) and O may be rescaled: PV(it - 1) must be done
            if (it > 0) {
                ok = wait_all(&bars.pv_done, (it - 1) & 1);
                if (!ok) break;
                tc::fence_after_sync();
            }
            if (__any_sync(0xffffffffu, over) && !w.first(t_begin)) {
                // rescale this row of O (earlier tiles of the unit)
#pragma unroll 1
                for (int c = 0; c < D; c += 16) {
                    uint32_t v[16];
                    tc::ld_32x32b_x16(lane_addr + 256 + c, v);
                    tc::wait_ld();
#pragma unroll
                    for (int e = 0; e < 16; ++e) v[e] = __float_as_uint(__uint_as_float(v[e]) * alpha);
                    tc::st_32x32b_x16(lane_addr + 256 + c, v);
                }
                tc::wait_st();
            }
            const float mu = m_used == -INFINITY ? 0.f : m_used;
#pragma unroll 1
            for (int c = 0; c < kTokTile; c += 16) {
                uint32_t v[16];
                tc::ld_32x32b_x16(s_addr + c, v);
                tc::wait_ld();
                uint32_t wd[8];
#pragma unroll
                for (int e = 0; e < 16; e += 2) {
                    const float p0 = c + e < vis ? ex2(fmaf(__uint_as_float(v[e]), a.scale_log2, -mu)) : 0.f;
                    const float p1 = c + e + 1 < vis ? ex2(fmaf(__uint_as_float(v[e + 1]), a.scale_log2, -mu)) : 0.f;
                    const __nv_bfloat162 h2 = __floats2bfloat162_rn(p0, p1);
                    l += __low2float(h2) + __high2float(h2);  // the weights P V uses
                    wd[e / 2] = *reinterpret_cast<const uint32_t *>(&h2);
                }
                // columns c .. c + 15 are 16-byte chunks 2 (c % 64) / 16, +1 of atom c / 64
                const int at = c >> 6, j0 = (c & 63) >> 3;
                *reinterpret_cast<uint4 *>(p_buf + at * kAtom + sw128(r, j0)) = make_uint4(wd[0], wd[1], wd[2], wd[3]);
                *reinterpret_cast<uint4 *>(p_buf + at * kAtom + sw128(r, j0 + 1)) = make_uint4(wd[4], wd[5], wd[6], wd[7]);
            }
            tc::fence_before_sync();
            __syncwarp();
            tc::mbar_arrive_elect(smem_u32(&bars.s_free[it & 1]));  // S(it) read
            tc::fence_proxy_async_smem();
            __syncwarp();
            tc::mbar_arrive_elect(smem_u32(&bars.p_full));
            if (w.last()) {
                // ---- the unit's partial: O / l and its log-sum-exp, slot u + part
                ok = wait_all(&bars.pv_done, it & 1);
                if (!ok) break;
                tc::fence_after_sync();
                const float inv = l > 0.f ? 1.f / l : 0.f;
                const int64_t slot = static_cast<int64_t>(u) + part;
                float *out = a.o_part + (slot * a.rows + r) * D;
#pragma unroll 1
                for (int c = 0; c < D; c += 16) {
                    uint32_t v[16];
                    tc::ld_32x32b_x16(lane_addr + 256 + c, v);
                    tc::wait_ld();
                    if (row_ok) {
#pragma unroll
                        for (int e = 0; e < 16; e += 4)
                            *reinterpret_cast<float4 *>(out + c + e) =
                                make_float4(__uint_as_float(v[e]) * inv, __uint_as_float(v[e + 1]) * inv,
                                            __uint_as_float(v[e + 2]) * inv, __uint_as_float(v[e + 3]) * inv);
                    }
                }
                if (row_ok)
                    a.lse_part[slot * a.rows + r] = l > 0.f ? (m_used + log2f(l)) * 0.69314718055994531f : -INFINITY;
                tc::fence_before_sync();
                __syncwarp();
            }
        }
        if (!ok && lane == 0) fail();
    }
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, 512);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode_gqa = nullptr;

cudaError_t encode_tile_map(CUtensorMap *m, const void *base, int cols, int64_t tok_stride, int64_t blk_stride,
                            int tokens_per_block, int blocks, int box_rows)
{
    if (!g_encode_gqa) {
        cudaDriverEntryPointQueryResult q;
        void *fn = nullptr;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return e != cudaSuccess ? e : cudaErrorNotSupported;
        g_encode_gqa = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(tokens_per_block),
                          static_cast<cuuint64_t>(blocks)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(tok_stride) * 2, static_cast<cuuint64_t>(blk_stride) * 2};
    cuuint32_t box[3] = {64, static_cast<cuuint32_t>(box_rows), 1}, es[3] = {1, 1, 1};
    CUresult r = g_encode_gqa(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
                              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <int D>
cudaError_t launch_d(const GqaLaunch &g, cudaStream_t st)
{
    const CacheView &c = g.cache;
    const bool paged = c.block_table != nullptr;
    const int tpb = paged ? c.page_size : c.capacity;
    const int blocks = paged ? c.num_pages : g.batch * g.groups;
    const int box_rows = paged ? 64 : kTokTile;
    CUtensorMap mk, mv;
    cudaError_t e;
    if ((e = encode_tile_map(&mk, c.k_rope, D, c.r_tok, c.r_blk, tpb, blocks, box_rows)) != cudaSuccess) return e;
    if ((e = encode_tile_map(&mv, c.c_kv, D, c.c_tok, c.c_blk, tpb, blocks, box_rows)) != cudaSuccess) return e;
    constexpr int tile = kTokTile * D * 2, atom = 128 * 128;
    int dev = 0, optin = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    const int fixed = 1024 + (D / 64) * atom + 2 * atom;
    const int static_bytes = static_cast<int>(sizeof(GqaBars)) + 64 * 8 + 64;
    int slots = (optin - static_bytes - fixed) / tile;
    if (slots > 2 * kMaxRing) slots = 2 * kMaxRing;
    if (slots < 2) return cudaErrorInvalidConfiguration;
    GqaArgs a;
    a.batch = g.batch;
    a.q_len = g.q_len;
    a.groups = g.groups;
    a.hpg = g.hpg;
    a.rows = g.q_len * g.hpg;
    a.max_kv = g.max_kv;
    a.num_splits = g.num_splits;
    a.paged = paged;
    a.bt_stride = c.bt_stride;
    a.num_pages = c.num_pages;
    a.nk = (slots + 1) / 2;
    a.nv = slots - a.nk;
    a.scale_log2 = g.sm_scale * 1.4426950408889634f;
    a.style = g.rope_style;
    a.kv_len = g.kv_len;
    a.block_table = c.block_table;
    a.q = static_cast<const uint16_t *>(g.q);
    a.o_part = g.o_part;
    a.lse_part = g.lse_part;
    a.status = g.status;
    a.turns = rope_turns(D, g.rope_base);
    const size_t smem = static_cast<size_t>(fixed) + static_cast<size_t>(slots) * tile;
    if ((e = cudaFuncSetAttribute(gqa_attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(smem))) != cudaSuccess)
        return e;
    return launch_dependent(gqa_attn_kernel<D>, dim3(1, g.num_splits, 1), dim3(kGqaThreads), smem, st, 1, a, mk, mv);
}

}  // namespace

cudaError_t launch_gqa_attn(const GqaLaunch &g, cudaStream_t st)
{
    if (g.batch <= 0) return cudaSuccess;
    if (g.q_len * g.hpg > 128) return cudaErrorInvalidConfiguration;
    if (g.head_dim == 64) return launch_d<64>(g, st);
    if (g.head_dim == 128) return launch_d<128>(g, st);
    return cudaErrorInvalidConfiguration;
}

}  // namespace gbmla
