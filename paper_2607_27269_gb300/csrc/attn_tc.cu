// Tensor-core split-KV attention core over the latent cache for sm_103a
// (Eqs. 2-4 with the Sec. 3.3 score routing, in the absorbed form).
//
// One CTA = (one partition of the tile list, one group of N query rows).  Per
// 128-token tile, with tokens on the MMA's M dimension and query rows on N:
//     S^T [128 tok, N] = [k_rope | c] tile (K-major A) x q_abs^T (K-major B)
//     online softmax over tokens (TMEM lane = token, column = query row)
//     O^T [r, N]      += C^T (latent tile read as an MN-major A) x P^T
// S^T (two buffers) and O^T live in TMEM.  The cache streams through two
// rings of 64-column chunks: the QK ring (positional keys, then the latent
// chunks of each tile) feeds the score products, the PV ring (the latent
// chunks again, from L2) the value products, so that the softmax of tile t
// overlaps QK(t+1) and PV(t-1).  More than 80 query rows run as several
// independent CTAs per partition, each loading the cache boxes itself (the
// later ones hit in L2).  A sequence's last, partial tile issues only
// the value products of its 16-token steps that hold cached rows; the PV warp
// clears the rows past the end inside the last such step itself.
//
// Warp roles (512 threads): warps 0 and 3 = TMA producers (QK ring and query
// boxes; PV ring), warp 1 = QK MMA issuer and TMEM owner, warp 2 = PV MMA
// issuer, warps 4..15 = softmax / epilogue (three warps per TMEM lane quarter,
// each owning every third 16-column block of the query columns).  Every wait
// is bounded; a wait that runs out records a timeout in the status word and
// the CTA winds down without trapping.
#include <cudaTypedefs.h>
#include <math.h>
#include <stdlib.h>

#include <type_traits>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace gbmla {
namespace {

constexpr int kTile = MLA_SPLIT_TILE;     // tokens per tile (MMA M)
constexpr int kHalf = 64;                 // tokens per TMA box (one page when paged)
constexpr int kChunkBytes = kTile * 128;  // 128 tokens x 64 bf16 columns, SW128 K-major
constexpr int kMaxSlots = 16;               // ring slots of both rings together
constexpr int kSoftmaxWarps = 12;
constexpr int kWhole = 1 << 30;             // flag bit beside a sequence index (batch < 2^30)
constexpr int kSoftmaxBase = 128;           // first softmax thread (after two producer and two MMA warps)
constexpr int kThreads = kSoftmaxBase + 32 * kSoftmaxWarps;

// P buffers: two, so that the softmax of tile t overlaps PV(t-1).  (With
// streamed queries an 80-row CTA has the room; with resident ones it then
// keeps only five ring slots.)
template <int N>
constexpr int kPBufs = 2;

// O^T buffers in TMEM: two where they fit beside the two S^T buffers (2N + 2 x 4N
// columns <= 512, i.e. N <= 48), so that a sequence's value products start in
// one while the previous sequence's partial drains from the other; else one.
template <int N>
constexpr int kOBufs = 10 * N <= 512 ? 2 : 1;
template <int N>
constexpr uint32_t kTmemCols = (2 * N + kOBufs<N> * 4 * N) <= 128 ? 128u
                               : (2 * N + kOBufs<N> * 4 * N) <= 256 ? 256u : 512u;


struct TcArgs {
    int batch, q_len, heads, rank, d_rope, rows, num_splits, max_kv;
    int paged, bt_stride, num_pages, qk_slots, pv_slots;
    float scale_log2;
    const int32_t *kv_len;
    const int32_t *block_table;
    float *o_part, *lse_part;
    // or NULL: a sequence whose tiles all lie in one partition writes its
    // (final) output and log-sum-exp here, at row b of [B, rows, ...], instead
    // of its partial slot (the combine then leaves that sequence alone)
    float *o_final, *lse_final;
    unsigned *status;
    uint64_t wait_ns;
};

struct __align__(8) Bars {
    uint64_t qk_full[kMaxSlots], qk_empty[kMaxSlots];  // QK ring: positional keys + latent chunks
    uint64_t pv_full[kMaxSlots], pv_empty[kMaxSlots];  // PV ring: latent chunks again
    uint64_t q_full, q_free;
    uint64_t s_full[2], s_free[2];
    uint64_t p_full[2], pv_done[2];  // per P buffer (t % NP): P(t) published / PV(t) completed
    uint64_t o_free, drain_qk, drain_pv;  // o_free: O^T buffer 0 drained
};

// With two O^T buffers, the barrier of the second.  (A kernel with one buffer
// keeps the plain layout: one more member there changed its register
// allocation enough to spill.)
struct BarsO2 : Bars {
    uint64_t o_free1;
};
template <int N>
using BarsT = std::conditional_t<kOBufs<N> == 2, BarsO2, Bars>;

template <class B>
__device__ __forceinline__ uint64_t *o_free_bar(B &b, int i)
{
    if constexpr (std::is_same_v<B, BarsO2>)
        return i ? &b.o_free1 : &b.o_free;
    else
        return &b.o_free;
}

template <int N>
struct Shared {
    float red[4][N];   // per TMEM-quadrant column partials
    float m_used[N];   // exponent base of each query column (log2 domain)
    float alpha[N];    // rescale factor of the current tile
    float lsum[N];     // softmax denominators at the epilogue (one O^T buffer)
    float inv_l[N];    // 1 / softmax denominator of the last closed sequence (two buffers)
    int lim[N];        // last visible position of each column (-1: padding column)
    int need_max;
    int any_rescale;
    int abort;         // any role gave up: producer / MMA stop issuing
    int sm_fail;       // softmax warps gave up (read only after a named barrier)
    uint32_t tmem_base;
};

// Tiles [t_begin, t_end) of the flattened tile list, sequence by sequence.
struct Walk {
    const int32_t *kv;
    int batch, q_len, max_kv;
    int b;
    int64_t seq_start, nb, t, t_begin, t_end;

    __device__ void init(const int32_t *kv_len, int batch_, int q_len_, int max_kv_, int64_t tb, int64_t te)
    {
        kv = kv_len;
        batch = batch_;
        q_len = q_len_;
        max_kv = max_kv_;
        t = tb;
        t_begin = tb;
        t_end = te;
        seq_start = 0;
        nb = 0;
        for (b = 0; b < batch; ++b) {
            nb = seq_tiles(kv[b], q_len, max_kv);
            if (seq_start + nb > t) break;
            seq_start += nb;
        }
    }
    __device__ bool done() const { return t >= t_end; }
    __device__ int tile() const { return static_cast<int>(t - seq_start); }
    __device__ bool first() const { return t == t_begin || t == seq_start; }
    __device__ bool last() const { return t + 1 == t_end || t + 1 == seq_start + nb; }
    __device__ bool last_of_partition() const { return t + 1 == t_end; }
    __device__ void next()
    {
        ++t;
        if (t < t_end && t >= seq_start + nb) {
            seq_start += nb;
            for (++b; b < batch; ++b) {
                nb = seq_tiles(kv[b], q_len, max_kv);
                if (nb > 0) break;
            }
        }
    }
};

// Where the boxes of tile j of sequence b live: a contiguous cache loads
// the tile as one 128-row box, a paged cache as one 64-row box per page.
struct TileLoc {
    int nh;            // boxes to load (0 if the first page is bad)
    uint32_t bytes;    // bytes the boxes deliver
    int32_t tok0[2], blk[2];
};

__device__ __forceinline__ TileLoc locate(const TcArgs &a, int b, int j)
{
    TileLoc L;
    if (!a.paged) {
        L.nh = 1;
        L.bytes = kTile * 128;
        L.blk[0] = b;
        L.tok0[0] = j * kTile;
        return L;
    }
    const int kv = a.kv_len[b];
    L.nh = (kv - j * kTile > kHalf) ? 2 : 1;
    for (int h = 0; h < L.nh; ++h) {
        const int32_t pg = a.block_table[static_cast<int64_t>(b) * a.bt_stride + 2 * j + h];
        if (pg < 0 || pg >= a.num_pages) {
            record_status(a.status, kStatusBounds);
            L.nh = h;
            break;
        }
        L.blk[h] = pg;
        L.tok0[h] = 0;
    }
    L.bytes = static_cast<uint32_t>(L.nh) * kHalf * 128;
    return L;
}

// A ring position: slot index and how many full passes over the ring came before.
struct RingPos {
    int slot, round;
    __device__ void advance(int cs)
    {
        if (++slot == cs) {
            slot = 0;
            ++round;
        }
    }
};

// Non-blocking test: has the phase with this parity completed?
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ void named_sync_softmax()
{
    asm volatile("bar.sync 1, %0;" ::"n"(32 * kSoftmaxWarps) : "memory");
}

// Reduce 16 columns over the 32 lanes of a warp: afterwards lane l holds, in
// v[0], the reduction of column (l % 16).
template <int CNT, bool MAX>
__device__ __forceinline__ void halve_step(float *v, int lane)
{
    const bool upper = (lane & CNT) != 0;
#pragma unroll
    for (int k = 0; k < CNT; ++k) {
        const float send = upper ? v[k] : v[k + CNT];
        const float keep = upper ? v[k + CNT] : v[k];
        const float recv = __shfl_xor_sync(0xffffffffu, send, CNT);
        v[k] = MAX ? fmaxf(keep, recv) : keep + recv;
    }
}

template <bool MAX>
__device__ __forceinline__ float reduce16(float (&v)[16], int lane)
{
#pragma unroll
    for (int k = 0; k < 16; ++k) {
        const float o = __shfl_xor_sync(0xffffffffu, v[k], 16);
        v[k] = MAX ? fmaxf(v[k], o) : v[k] + o;
    }
    halve_step<8, MAX>(v, lane);
    halve_step<4, MAX>(v, lane);
    halve_step<2, MAX>(v, lane);
    halve_step<1, MAX>(v, lane);
    return v[0];
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    tc::ld_32x32b_x16(taddr, r);
    tc::wait_ld();
#pragma unroll
    for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(r[j]);
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float (&v)[16])
{
    uint32_t r[16];
#pragma unroll
    for (int j = 0; j < 16; ++j) r[j] = __float_as_uint(v[j]);
    tc::st_32x32b_x16(taddr, r);
    tc::wait_st();
}

// Where sequence b's output rows and log-sum-exps go: its partial slot b + k,
// or (whole: all its tiles in this partition, and a final buffer given) its
// final row b.
__device__ __forceinline__ float *out_rows(const TcArgs &a, int b, int part, bool whole)
{
    return whole && a.o_final ? a.o_final + static_cast<int64_t>(b) * a.rows * a.rank
                              : a.o_part + (static_cast<int64_t>(b) + part) * a.rows * a.rank;
}

__device__ __forceinline__ float *lse_rows(const TcArgs &a, int b, int part, bool whole)
{
    return whole && a.lse_final ? a.lse_final + static_cast<int64_t>(b) * a.rows
                                : a.lse_part + (static_cast<int64_t>(b) + part) * a.rows;
}

// Per-thread constants of a softmax warp.
struct SmCtx {
    int lane, tid, quarter, half, tok, n_own, group, part, nrc, ncc, cs, n_items;
    uint32_t lane_base, tmem, o_col0;
    unsigned char *ring, *p_buf;  // p_buf: NP buffers of NB x [128 tok x 32 B]
    uint64_t lim_ns;
    int64_t t_begin, t_end;
};

// The whole warp waits; a failure marks sm_fail, which the softmax
// warps read only after their next named barrier, so they all leave together.
template <int N>
__device__ __forceinline__ void sm_wait(const SmCtx &c, const TcArgs &a, Shared<N> &ss, uint64_t *bar,
                                        uint32_t parity)
{
    if (!__all_sync(0xffffffffu, mbar_wait(smem_u32(bar), parity, c.lim_ns)) && c.lane == 0) {
        record_status(a.status, kStatusTimeout);
        atomicOr(&ss.sm_fail, 1);
        ss.abort = 1;
    }
    __syncwarp();
}

// Scores of one 16-column block in the log2 domain, masked where needed.
template <int N>
__device__ __forceinline__ void sm_scores(const TcArgs &a, const Shared<N> &ss, uint32_t s_base, int cb, int pos,
                                          bool need_mask, float (&s)[16])
{
    tmem_ld16(s_base + cb * 16, s);
#pragma unroll
    for (int e = 0; e < 16; ++e) {
        s[e] *= a.scale_log2;
        if (need_mask && pos > ss.lim[cb * 16 + e]) s[e] = -INFINITY;
    }
}

// Column maxima of the tile's scores over this warp's 32 tokens, into red[quarter].
template <int N, int KOWN>
__device__ __forceinline__ void sm_block_max(const SmCtx &c, const TcArgs &a, Shared<N> &ss, uint32_t s_base,
                                             int pos, bool need_mask)
{
#pragma unroll
    for (int ob = 0; ob < KOWN; ++ob) {
        if (ob < c.n_own) {
            const int cb = c.half + 3 * ob;
            float s[16];
            sm_scores<N>(a, ss, s_base, cb, pos, need_mask, s);
            const float mx = reduce16<true>(s, c.lane);
            if (c.lane < 16) ss.red[c.quarter][cb * 16 + c.lane] = mx;
        }
    }
}

// Normalised partial output and log-sum-exp of sequence b, whose last tile
// in this partition was t_end_seg, in one step (one O^T buffer).
template <int N, int KOWN>
__device__ __forceinline__ void sm_epilogue(const SmCtx &c, const TcArgs &a, Shared<N> &ss, Bars &bars,
                                            float (&l_part)[KOWN][16], int b, int64_t t_end_seg, bool whole)
{
    sm_wait<N>(c, a, ss, &bars.pv_done[t_end_seg % kPBufs<N>], static_cast<uint32_t>((t_end_seg / kPBufs<N>) & 1));
    named_sync_softmax();
    if (ss.sm_fail) return;
    tc::fence_after_sync();
#pragma unroll
    for (int ob = 0; ob < KOWN; ++ob) {
        if (ob < c.n_own) {
            const int cb = c.half + 3 * ob;
            float v[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) v[e] = l_part[ob][e];
            const float ls = reduce16<false>(v, c.lane);
            if (c.lane < 16) ss.red[c.quarter][cb * 16 + c.lane] = ls;
        }
    }
    named_sync_softmax();
    const int cc = c.tid - kSoftmaxBase;
    if (cc < N) {
        const float l = ss.red[0][cc] + ss.red[1][cc] + ss.red[2][cc] + ss.red[3][cc];
        ss.lsum[cc] = l;
        ss.alpha[cc] = l > 0.f ? 1.f / l : 0.f;  // reused here as 1 / l
    }
    named_sync_softmax();
    const int valid_cols = a.rows - c.group * N;  // columns past it are padding
    float *out = out_rows(a, b, c.part, whole) + static_cast<int64_t>(c.group) * N * a.rank + c.tok;
    for (int m = 0; m < c.nrc; ++m) {
#pragma unroll
        for (int ob = 0; ob < KOWN; ++ob) {
            if (ob < c.n_own) {
                const int cb = c.half + 3 * ob;
                float o[16];
                tmem_ld16(c.tmem + c.lane_base + c.o_col0 + m * N + cb * 16, o);
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int col = cb * 16 + e;
                    if (col < valid_cols) out[col * a.rank + m * 128] = o[e] * ss.alpha[col];
                }
            }
        }
    }
    if (cc < N) {
        const int row = c.group * N + cc;
        if (row < a.rows) {
            const float l = ss.lsum[cc];
            lse_rows(a, b, c.part, whole)[row] = l > 0.f ? (ss.m_used[cc] + log2f(l)) * 0.69314718055994531f : -INFINITY;
        }
    }
    tc::fence_before_sync();
    __syncwarp();
    if (c.lane == 0) tc::mbar_arrive(smem_u32(&bars.o_free));
}

// Closing a sequence b of this partition (no wait on its value products):
// its softmax denominators (1 / l kept for the drain) and its log-sum-exp.
template <int N, int KOWN>
__device__ __forceinline__ void sm_close(const SmCtx &c, const TcArgs &a, Shared<N> &ss, float (&l_part)[KOWN][16],
                                         int b, bool whole)
{
#pragma unroll
    for (int ob = 0; ob < KOWN; ++ob) {
        if (ob < c.n_own) {
            const int cb = c.half + 3 * ob;
            float v[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) v[e] = l_part[ob][e];
            const float ls = reduce16<false>(v, c.lane);
            if (c.lane < 16) ss.red[c.quarter][cb * 16 + c.lane] = ls;
        }
    }
    named_sync_softmax();
    const int cc = c.tid - kSoftmaxBase;
    if (cc < N) {
        const float l = ss.red[0][cc] + ss.red[1][cc] + ss.red[2][cc] + ss.red[3][cc];
        ss.inv_l[cc] = l > 0.f ? 1.f / l : 0.f;
        const int row = c.group * N + cc;
        if (row < a.rows)
            lse_rows(a, b, c.part, whole)[row] = l > 0.f ? (ss.m_used[cc] + log2f(l)) * 0.69314718055994531f : -INFINITY;
    }
    named_sync_softmax();  // inv_l is complete and red is free again
}

// The normalised partial output of sequence b (closed by sm_close), whose
// last tile here was t_end_seg, from O^T buffer obuf; then the buffer is free.
template <int N, int KOWN>
__device__ __forceinline__ void sm_drain(const SmCtx &c, const TcArgs &a, Shared<N> &ss, BarsT<N> &bars, int b,
                                         int64_t t_end_seg, int obuf, bool whole)
{
    sm_wait<N>(c, a, ss, &bars.pv_done[t_end_seg % kPBufs<N>], static_cast<uint32_t>((t_end_seg / kPBufs<N>) & 1));
    named_sync_softmax();
    if (ss.sm_fail) return;
    tc::fence_after_sync();
    const int valid_cols = a.rows - c.group * N;  // columns past it are padding
    float *out = out_rows(a, b, c.part, whole) + static_cast<int64_t>(c.group) * N * a.rank + c.tok;
    const uint32_t o_col = c.o_col0 + static_cast<uint32_t>(obuf * 4 * N);
    for (int m = 0; m < c.nrc; ++m) {
#pragma unroll
        for (int ob = 0; ob < KOWN; ++ob) {
            if (ob < c.n_own) {
                const int cb = c.half + 3 * ob;
                float o[16];
                tmem_ld16(c.tmem + c.lane_base + o_col + m * N + cb * 16, o);
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int col = cb * 16 + e;
                    if (col < valid_cols) out[col * a.rank + m * 128] = o[e] * ss.inv_l[col];
                }
            }
        }
    }
    tc::fence_before_sync();
    __syncwarp();
    if (c.lane == 0) tc::mbar_arrive(smem_u32(o_free_bar(bars, obuf)));
}

template <int N>
__device__ __forceinline__ void softmax_role(const SmCtx &c, const TcArgs &a, Shared<N> &ss, BarsT<N> &bars)
{
    constexpr int NB = N / 16;
    constexpr int KOWN = (NB + 2) / 3;
    float l_part[KOWN][16];
    // the sequence open here, with kWhole set when all its tiles lie in this
    // partition (its rows then go to the final buffers, when given)
    int b_cur = -1;
    int u = -1;  // sequences begun here (the PV warp counts the same ones)
    int64_t t_prev = -1;  // the previous tile (one O^T buffer: the drain runs at the next sequence's first tile)
    // a closed sequence whose drain waits for the next sequence's first P (two O^T buffers)
    int d_b = -1, d_t = -1;
    const int cc = c.tid - kSoftmaxBase;
    Walk w;
    w.init(a.kv_len, a.batch, a.q_len, a.max_kv, c.t_begin, c.t_end);
    for (int64_t t = 0; !w.done(); ++t, w.next()) {
        const bool first = w.first(), last = w.last();
        const int b = w.b, j = w.tile();
        const int kv = a.kv_len[b];
        const int sb = static_cast<int>(t & 1);
        sm_wait<N>(c, a, ss, &bars.s_full[sb], static_cast<uint32_t>((t >> 1) & 1));
        named_sync_softmax();
        if (ss.sm_fail) break;
        tc::fence_after_sync();
        if (first) {
            if constexpr (kOBufs<N> == 1) {
                if (b_cur >= 0) {
                    sm_epilogue<N, KOWN>(c, a, ss, bars, l_part, b_cur & ~kWhole, t_prev, (b_cur & kWhole) != 0);
                    if (ss.sm_fail) break;
                }
            }
            b_cur = b | (w.seq_start >= w.t_begin && w.seq_start + w.nb <= w.t_end ? kWhole : 0);
            ++u;
#pragma unroll
            for (int ob = 0; ob < KOWN; ++ob)
#pragma unroll
                for (int e = 0; e < 16; ++e) l_part[ob][e] = 0.f;
            if (cc < N) {
                const int row = c.group * N + cc;
                ss.lim[cc] = row < a.rows ? kv - a.q_len + row / a.heads : -1;
            }
            named_sync_softmax();
        }
        t_prev = t;
        const int pos = j * kTile + c.tok;
        // the mask matters only where a token lies past the earliest query's last key
        const bool need_mask = j * kTile + kTile - 1 > kv - a.q_len;
        const uint32_t s_base = c.tmem + c.lane_base + sb * N;
        // ---- pass 1: exponent bases (exact column maxima on a sequence's first
        // tile, else only when a score passes the current base by more than 2^8)
        if (first) {
            sm_block_max<N, KOWN>(c, a, ss, s_base, pos, need_mask);
            named_sync_softmax();
            if (cc < N) {
                ss.m_used[cc] = fmaxf(fmaxf(ss.red[0][cc], ss.red[1][cc]), fmaxf(ss.red[2][cc], ss.red[3][cc]));
                ss.alpha[cc] = 1.f;
            }
            if (c.tid == kSoftmaxBase) ss.any_rescale = 0;
        } else {
            bool over = false;
#pragma unroll
            for (int ob = 0; ob < KOWN; ++ob) {
                if (ob < c.n_own) {
                    const int cb = c.half + 3 * ob;
                    float s[16];
                    sm_scores<N>(a, ss, s_base, cb, pos, need_mask, s);
#pragma unroll
                    for (int e = 0; e < 16; ++e) over |= s[e] > ss.m_used[cb * 16 + e] + 8.f;
                }
            }
            if (__any_sync(0xffffffffu, over) && c.lane == 0) ss.need_max = 1;
            named_sync_softmax();
            if (ss.need_max) {  // uniform: written before the barrier, read after it
                sm_block_max<N, KOWN>(c, a, ss, s_base, pos, need_mask);
                named_sync_softmax();
                if (cc < N) {
                    const float tmax = fmaxf(fmaxf(ss.red[0][cc], ss.red[1][cc]), fmaxf(ss.red[2][cc], ss.red[3][cc]));
                    const float m_old = ss.m_used[cc];
                    float alpha = 1.f;
                    if (tmax != -INFINITY && (m_old == -INFINITY || tmax > m_old + 8.f)) {
                        alpha = m_old == -INFINITY ? 0.f : exp2f(m_old - tmax);
                        ss.m_used[cc] = tmax;
                    }
                    ss.alpha[cc] = alpha;
                }
                if (c.tid == kSoftmaxBase) {
                    ss.any_rescale = 1;
                    ss.need_max = 0;
                }
            } else if (c.tid == kSoftmaxBase) {
                ss.any_rescale = 0;
            }
        }
        named_sync_softmax();
        // ---- P(t) goes to buffer t % NP, free again once PV(t - NP) has
        // completed; O^T is rescaled (rarely: only when a base moves) once
        // PV(t-1) has completed.  Each wait is on the next phase of its barrier.
        constexpr int NP = kPBufs<N>;
        if (t >= NP) sm_wait<N>(c, a, ss, &bars.pv_done[t % NP], static_cast<uint32_t>(((t - NP) / NP) & 1));
        if (ss.any_rescale)  // never on a sequence's first tile
            sm_wait<N>(c, a, ss, &bars.pv_done[(t - 1) % NP], static_cast<uint32_t>(((t - 1) / NP) & 1));
        named_sync_softmax();
        if (ss.sm_fail) break;
        tc::fence_after_sync();
        {
            if (ss.any_rescale) {
#pragma unroll
                for (int ob = 0; ob < KOWN; ++ob) {
                    if (ob < c.n_own) {
                        const int cb = c.half + 3 * ob;
                        float al[16];
#pragma unroll
                        for (int e = 0; e < 16; ++e) {
                            al[e] = ss.alpha[cb * 16 + e];
                            l_part[ob][e] *= al[e];
                        }
                        for (int m = 0; m < c.nrc; ++m) {
                            const uint32_t ta = c.tmem + c.lane_base + c.o_col0 +
                                                static_cast<uint32_t>((u % kOBufs<N>) * 4 * N + m * N + cb * 16);
                            float o[16];
                            tmem_ld16(ta, o);
#pragma unroll
                            for (int e = 0; e < 16; ++e) o[e] *= al[e];
                            tmem_st16(ta, o);
                        }
                    }
                }
            }
        }
        // ---- pass 2: P = 2^(s - m) in bf16 (MN-major, 16-column SW32 atoms), running sums
#pragma unroll
        for (int ob = 0; ob < KOWN; ++ob) {
            if (ob < c.n_own) {
                const int cb = c.half + 3 * ob;
                float s[16];
                sm_scores<N>(a, ss, s_base, cb, pos, need_mask, s);
                uint32_t pk[8];
#pragma unroll
                for (int e = 0; e < 16; e += 2) {
                    const float p0 = s[e] == -INFINITY ? 0.f : exp2f(s[e] - ss.m_used[cb * 16 + e]);
                    const float p1 = s[e + 1] == -INFINITY ? 0.f : exp2f(s[e + 1] - ss.m_used[cb * 16 + e + 1]);
                    const __nv_bfloat162 pb = __floats2bfloat162_rn(p0, p1);
                    l_part[ob][e] += __low2float(pb);  // the weights the MMA multiplies by
                    l_part[ob][e + 1] += __high2float(pb);
                    pk[e / 2] = *reinterpret_cast<const uint32_t *>(&pb);
                }
                unsigned char *row = c.p_buf + (t % kPBufs<N>) * (N / 16) * (kTile * 32) + cb * (kTile * 32) + c.tok * 32;
                const int sw = (c.tok >> 2) & 1;
                *reinterpret_cast<uint4 *>(row + (sw * 16)) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
                *reinterpret_cast<uint4 *>(row + ((1 ^ sw) * 16)) = make_uint4(pk[4], pk[5], pk[6], pk[7]);
            }
        }
        tc::fence_before_sync();
        __syncwarp();
        if (c.lane == 0) tc::mbar_arrive(smem_u32(&bars.s_free[sb]));
        tc::fence_proxy_async_smem();
        tc::fence_before_sync();
        __syncwarp();
        if (c.lane == 0) tc::mbar_arrive(smem_u32(&bars.p_full[t % kPBufs<N>]));
        if constexpr (kOBufs<N> == 2) {
            // Due now, in this order: the previous sequence's drain (deferred
            // until this first P was out, so that it overlaps this tile's value
            // products in the other O^T buffer); then, on a sequence's last
            // tile, its close -- and at the partition's end its drain.
#pragma unroll 1
            for (int k = 0; k < 2; ++k) {
                int db = -1, dt = 0, dbuf = 0;
                if (k == 0 && d_b >= 0) {
                    db = d_b;
                    dt = d_t;
                    dbuf = (u - 1) & 1;
                    d_b = -1;
                }
                if (k == 1 && last) {
                    named_sync_softmax();
                    sm_close<N, KOWN>(c, a, ss, l_part, b_cur & ~kWhole, (b_cur & kWhole) != 0);
                    if (!w.last_of_partition()) {
                        d_b = b_cur;
                        d_t = static_cast<int>(t);
                    } else {
                        db = b_cur;
                        dt = static_cast<int>(t);
                        dbuf = u & 1;
                    }
                    b_cur = -1;
                }
                if (db >= 0) {
                    named_sync_softmax();
                    sm_drain<N, KOWN>(c, a, ss, bars, db & ~kWhole, dt, dbuf, (db & kWhole) != 0);
                    if (ss.sm_fail) break;
                }
            }
            if (ss.sm_fail) break;
        }
    }
    named_sync_softmax();
    if constexpr (kOBufs<N> == 1) {
        if (b_cur >= 0 && !ss.sm_fail)
            sm_epilogue<N, KOWN>(c, a, ss, bars, l_part, b_cur & ~kWhole, t_prev, (b_cur & kWhole) != 0);
    }
}

// N: query rows per CTA (multiple of 16, <= 80).  SQ (streamed queries): no
// resident query buffer; each QK-ring slot holds a cache chunk and, behind it,
// the query chunk that multiplies it, loaded with it from L2.  The ring then
// gets the shared memory the resident queries held, so that more cache bytes
// are in flight per SM, at the price of re-reading the queries once per tile.
template <int N, bool SQ>
__global__ void __maxnreg__(128)
    attn_tc_kernel(const __grid_constant__ TcArgs a, const __grid_constant__ CUtensorMap map_c,
                   const __grid_constant__ CUtensorMap map_r, const __grid_constant__ CUtensorMap map_q)
{
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ BarsT<N> bars;
    __shared__ Shared<N> ss;
    __shared__ int64_t red64[32];

    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~static_cast<uintptr_t>(1023));
    const int ncc = a.rank / 64;    // latent chunks per tile
    const int nrc = a.rank / 128;   // r-chunks of O^T
    const int nqc = ncc + 1;        // chunks of a tile in the QK pass: positional keys, then latent
    const int CA = a.qk_slots;      // QK ring slots
    const int CB = a.pv_slots;      // PV ring slots (even)
    static_assert(!SQ || (N * 128) % 1024 == 0, "a streamed query chunk keeps the slots 1024-byte aligned");
    constexpr int kSlotA = SQ ? kChunkBytes + N * 128 : kChunkBytes;       // QK-ring slot
    unsigned char *q_buf = smem;                                          // nqc x [N x 128 B] (resident queries)
    unsigned char *ring_a = SQ ? smem : q_buf + ((nqc * N * 128 + 1023) & ~1023);  // CA x [kSlotA]
    unsigned char *ring_b = ring_a + CA * kSlotA;                         // CB x [128 x 128 B]
    unsigned char *p_buf = ring_b + CB * kChunkBytes;                     // NP x NB x [128 tok x 32 B]

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int group = blockIdx.x, part = blockIdx.y;
    const uint64_t lim_ns = a.wait_ns;

    if (tid == 0) {
        for (int i = 0; i < kMaxSlots; ++i) {
            mbar_init(&bars.qk_full[i], 1);
            mbar_init(&bars.qk_empty[i], 1);
            mbar_init(&bars.pv_full[i], 1);
            mbar_init(&bars.pv_empty[i], 1);
        }
        mbar_init(&bars.q_full, 1);
        mbar_init(&bars.q_free, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars.s_full[i], 1);
            mbar_init(&bars.s_free[i], kSoftmaxWarps);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars.p_full[i], kSoftmaxWarps);
            mbar_init(&bars.pv_done[i], 1);
        }
        mbar_init(&bars.o_free, kSoftmaxWarps);
        if constexpr (kOBufs<N> == 2) mbar_init(o_free_bar(bars, 1), kSoftmaxWarps);
        mbar_init(&bars.drain_qk, 1);
        mbar_init(&bars.drain_pv, 1);
        ss.need_max = 0;
        ss.any_rescale = 0;
        ss.abort = 0;
        ss.sm_fail = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(smem_u32(&ss.tmem_base), kTmemCols<N>);
        tc::tmem_relinquish();
    }
    tc::fence_before_sync();
    __syncthreads();
    tc::fence_after_sync();
    // The queries come from the previous launch; the cache does not: every
    // kernel of this library that writes the cache (append, projection) lets
    // its dependents launch only once it has completed, so by the time this
    // kernel runs (launched by its predecessor's trigger, which follows the
    // predecessor's own wait) the cache is final.  So no thread waits here:
    // the TMA producers load cache tiles at once, the query lanes wait before
    // the first query load and the softmax warps before they write partials
    // (a predecessor may still read the partial buffers); the MMA warps touch
    // only shared and tensor memory.
    griddep_launch_dependents();

    if (part == 0 && group == 0) {
        for (int bb = tid; bb < a.batch; bb += kThreads) {
            const int kv = a.kv_len[bb];
            if (kv < a.q_len || kv > a.max_kv) record_status(a.status, kStatusBounds);
        }
    }
    const int64_t T = block_tile_sum(a.kv_len, a.batch, a.q_len, a.max_kv, red64);
    const int64_t t_begin = T ? part_begin(part, T, a.num_splits) : 0;
    const int64_t t_end = T ? part_begin(part + 1, T, a.num_splits) : 0;
    const int n_items = static_cast<int>(t_end - t_begin);
    const uint32_t tmem = ss.tmem_base;
    const uint32_t o_col0 = 2 * N;   // S^T buffers at columns [0, N) and [N, 2N); O^T buffer i at 2N + 4N i
    auto any_abort = [&]() {
        return __any_sync(0xffffffffu, *reinterpret_cast<volatile int *>(&ss.abort) != 0);
    };

    if (warp == 0 || warp == 3) {
        // ================================================================ TMA producers
        // A tensor-TMA instruction occupies its issuing thread for a long,
        // nearly size-independent time, so the loads are spread over lanes
        // and warps, each lane an independent in-order stream.  Warp 0: lane
        // s < CA refills QK-ring slot s (chunks s, s + CA, ... of the QK pass,
        // nqc per tile: positional keys, then the latent chunks) -- with
        // streamed queries the chunk's cache box(es) and then its query box
        // (the first pass's query box waits for the next pass, after
        // griddepcontrol.wait); with resident queries lanes 16..16+ncc load
        // the query boxes of each sequence.  Warp 3: lane s < CB refills
        // PV-ring slot s (chunks s, s + CB, ... of the PV pass, ncc per
        // tile).  The lanes of a warp poll their own barrier without
        // blocking in one converged loop, and every lane whose slot is free
        // issues in the same pass.  A lane waits only on phases of its own
        // barrier, in order, so every parity test is on the next phase.
        if (n_items > 0) {
            if (lane == 0 && warp == 0) {
                tc::prefetch_tensormap(&map_c);
                tc::prefetch_tensormap(&map_r);
                tc::prefetch_tensormap(&map_q);
            }
            enum { kQK, kPV, kQuery, kIdle };
            const int kind = warp == 3 ? (lane < CB ? kPV : kIdle)
                                       : (lane < CA ? kQK : (!SQ && lane >= 16 && lane < 16 + nqc) ? kQuery : kIdle);
            const int slot = lane;
            const int per_tile = kind == kQK ? nqc : ncc;
            const int ring_len = kind == kQK ? CA : CB;
            Walk w;
            w.init(a.kv_len, a.batch, a.q_len, a.max_kv, t_begin, t_end);
            const int64_t total = static_cast<int64_t>(n_items) * per_tile;
            int64_t c = slot;  // ring lanes: next chunk of this lane's pass
            int64_t k = 0;     // jobs this lane has issued (ring round / sequence)
            bool has = (kind == kQK || kind == kPV) ? c < total : kind == kQuery;
            bool ok = true;
            uint64_t wait_t0 = 0;
            // griddepcontrol.wait still to do before the first query load
            bool q_pending = SQ ? kind == kQK : kind == kQuery;
            // streamed queries: the query box of the chunk issued in the first
            // pass, which waits for that pass's griddepcontrol.wait
            bool q_owed = false;
            int q_owed_x = 0, q_owed_y = 0;
            bool first_pass = true;           // the ring lanes issue their first cache loads in it
            const uint64_t pol_keep = tc::policy_evict_last(), pol_drop = tc::policy_evict_first();
            uint32_t wbar = 0, fbar = 0, dst = 0;
            if (kind == kQK) {
                wbar = smem_u32(&bars.qk_empty[slot]);
                fbar = smem_u32(&bars.qk_full[slot]);
                dst = smem_u32(ring_a + slot * kSlotA);
            } else if (kind == kPV) {
                wbar = smem_u32(&bars.pv_empty[slot]);
                fbar = smem_u32(&bars.pv_full[slot]);
                dst = smem_u32(ring_b + slot * kChunkBytes);
            } else if (kind == kQuery) {
                wbar = smem_u32(&bars.q_free);
                fbar = smem_u32(&bars.q_full);
                dst = smem_u32(q_buf + (lane - 16) * N * 128);
            }
            while (true) {
                if (kind == kQuery) has = has && !w.done();
                if (!__any_sync(0xffffffffu, (has || q_owed) && ok)) break;
                if (any_abort()) break;
                bool progressed = false;
                if (q_pending && !first_pass) {
                    griddep_wait();
                    q_pending = false;
                    if (SQ && q_owed) {
                        tc::tma_load_2d_hint(dst + kChunkBytes, &map_q, q_owed_x, q_owed_y, fbar, pol_keep);
                        q_owed = false;
                        progressed = true;
                    }
                }
                if (has && ok && !(kind == kQuery && q_pending)) {
                    const bool ready = k == 0 || mbar_test(wbar, static_cast<uint32_t>((k - 1) & 1));
                    if (!ready) {
                        const uint64_t now = global_ns();
                        if (wait_t0 == 0)
                            wait_t0 = now;
                        else if (now - wait_t0 > lim_ns)
                            ok = false;
                    } else {
                        wait_t0 = 0;
                        progressed = true;
                        if (kind == kQuery) {
                            const int box = lane - 16;
                            if (box == 0) tc::mbar_arrive_expect_tx(fbar, nqc * N * 128);
                            tc::tma_load_2d(dst, &map_q, 64 * box, w.b * a.rows + group * N, fbar);
                            do {
                                w.next();
                            } while (!w.done() && !w.first());
                        } else {
                            const int64_t tile = c / per_tile;
                            const int i = static_cast<int>(c - tile * per_tile);
                            while (w.t < t_begin + tile) w.next();
                            const TileLoc L = locate(a, w.b, w.tile());
                            // QK pass: chunk 0 = positional keys, 1.. = latent; PV pass: latent
                            const bool keys = kind == kQK && i == 0;
                            const CUtensorMap *map = keys ? &map_r : &map_c;
                            const int col = keys ? 0 : 64 * (kind == kQK ? i - 1 : i);
                            const bool sq = SQ && kind == kQK;
                            tc::mbar_arrive_expect_tx(fbar, L.bytes + (sq ? N * 128 : 0));
                            // the QK pass keeps latent lines in L2 for the PV pass, which reads
                            // them a last time; the positional keys are read once
                            const uint64_t pol = (kind == kQK && !keys) ? pol_keep : pol_drop;
                            for (int h = 0; h < L.nh; ++h)
                                tc::tma_load_3d_hint(dst + h * kHalf * 128, map, col, L.tok0[h], L.blk[h], fbar,
                                                     pol);
                            if (sq) {
                                // the query columns this chunk multiplies: the positional
                                // part behind the latent part in each query row
                                const int qx = 64 * (keys ? ncc : i - 1);
                                const int qy = w.b * a.rows + group * N;
                                if (q_pending) {
                                    q_owed = true;
                                    q_owed_x = qx;
                                    q_owed_y = qy;
                                } else {
                                    tc::tma_load_2d_hint(dst + kChunkBytes, &map_q, qx, qy, fbar, pol_keep);
                                }
                            }
                            c += ring_len;
                            has = c < total;
                        }
                        ++k;
                    }
                }
                if (!__any_sync(0xffffffffu, progressed)) __nanosleep(32);
                first_pass = false;
            }
            if (q_pending) griddep_wait();  // (no query was loaded: keep the wait before leaving)
            if (!ok) {
                record_status(a.status, kStatusTimeout);
                ss.abort = 1;
            }
            __syncwarp();
        }
    } else if (warp == 1 || warp == 2) {
        // ================================================================ MMA issuers
        // Warp 1 issues the score products QK(t), warp 2 the value products
        // PV(t); each consumes its own ring in order.  The whole warp runs its
        // loop converged (every lane waits); one elected lane issues each MMA,
        // commit and arrive.
        const bool is_qk = warp == 1;
        uint64_t *drain = is_qk ? &bars.drain_qk : &bars.drain_pv;
        if (n_items > 0) {
            const uint32_t q_base = smem_u32(q_buf), p_base = smem_u32(p_buf);
            // descriptor templates (start address added per MMA)
            const uint64_t dq = tc::smem_desc(0, 16, 1024, tc::kSwizzle128B);
            const uint64_t dc = tc::smem_desc(0, kChunkBytes, 1024, tc::kSwizzle128B);
            const uint64_t dp = tc::smem_desc(0, 128 * 32, 256, tc::kSwizzle32B);
            auto with_addr = [](uint64_t tmpl, uint32_t saddr) {
                return tmpl | static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
            };
            Walk w;
            w.init(a.kv_len, a.batch, a.q_len, a.max_kv, t_begin, t_end);
            RingPos rp{0, 0};
            bool ok = true;
            auto wait = [&](uint64_t *bar, uint32_t parity) {
                if (ok) ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(bar), parity, lim_ns));
                return ok;
            };
            // a consumed slot is handed back to its producer lane
            auto release = [&](uint64_t *bar) { tc::commit_elect(smem_u32(bar)); };
            if (is_qk) {
                const uint32_t id_qk = tc::idesc_bf16_f32(128, N, false, false);
                const uint32_t ring_base = smem_u32(ring_a);
                int seg = -1;
                for (int t = 0; t < n_items && ok; ++t, w.next()) {
                    if (any_abort()) break;
                    if (!SQ && w.first()) {
                        ++seg;
                        if (!wait(&bars.q_full, seg & 1)) break;
                    }
                    const int sb = t & 1;
                    if (t >= 2 && !wait(&bars.s_free[sb], ((t >> 1) - 1) & 1)) break;
                    const uint32_t d_s = tmem + sb * N;
                    for (int i = 0; i < nqc && ok; ++i) {
                        if (!wait(&bars.qk_full[rp.slot], rp.round & 1)) break;
                        tc::fence_after_sync();
                        const uint32_t cb = ring_base + rp.slot * kSlotA;
                        const uint32_t qb = SQ ? cb + kChunkBytes : q_base + (i == 0 ? ncc : i - 1) * N * 128;
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            tc::mma_bf16_elect(d_s, with_addr(dq, cb + kk * 32), with_addr(dq, qb + kk * 32), id_qk,
                                               (i | kk) != 0);
                        release(&bars.qk_empty[rp.slot]);
                        rp.advance(CA);
                    }
                    if (!ok) break;
                    tc::commit_elect(smem_u32(&bars.s_full[sb]));
                    if (!SQ && w.last()) tc::commit_elect(smem_u32(&bars.q_free));
                }
            } else {
                const uint32_t id_pv = tc::idesc_bf16_f32(128, N, true, true);
                const uint32_t ring_base = smem_u32(ring_b);
                int seg = -1;
                uint32_t o_cur = o_col0;
                for (int t = 0; t < n_items && ok; ++t, w.next()) {
                    if (any_abort()) break;
                    if (!wait(&bars.p_full[t % kPBufs<N>], (t / kPBufs<N>) & 1)) break;
                    bool first_pv = false;
                    if (w.first()) {
                        // buffer seg % kOBufs: wait until the sequence that used it last has drained
                        ++seg;
                        const int ob = seg % kOBufs<N>, use = seg / kOBufs<N>;
                        if (use >= 1 && !wait(o_free_bar(bars, ob), (use - 1) & 1)) break;
                        o_cur = o_col0 + static_cast<uint32_t>(ob * 4 * N);
                        first_pv = true;
                    }
                    // A sequence's last, partial tile of v rows: only the 16-token
                    // steps holding rows < v are issued, and in the last of them the
                    // rows v .. v16 - 1 of both chunks are cleared here first, so that
                    // stale or uninitialised bytes never meet a zero weight (0 x NaN
                    // is NaN).  Rows past v16 are never read.
                    const int v = a.kv_len[w.b] - w.tile() * kTile;
                    const bool tail = w.last() && v < kTile;
                    const int v16 = tail ? (v + 15) / 16 * 16 : kTile;
                    for (int m = 0; m < nrc && ok; ++m) {
                        // chunks 2m, 2m+1 sit in adjacent slots (CB and ncc are even)
                        const int s0 = rp.slot;
                        if (!wait(&bars.pv_full[s0], rp.round & 1) || !wait(&bars.pv_full[s0 + 1], rp.round & 1)) break;
                        tc::fence_after_sync();
                        if (v16 > v) {
                            const int nz = (v16 - v) * 8;  // 16-byte pieces per chunk
                            for (int idx = lane; idx < 2 * nz; idx += 32) {
                                const int k = idx / nz, r = idx - k * nz;
                                uint4 *dst = reinterpret_cast<uint4 *>(ring_b + (s0 + k) * kChunkBytes +
                                                                       (v + r / 8) * 128) + r % 8;
                                *dst = make_uint4(0, 0, 0, 0);
                            }
                            tc::fence_proxy_async_smem();
                            __syncwarp();
                        }
                        const uint32_t cb = ring_base + s0 * kChunkBytes;
                        const uint32_t pb = p_base + (t % kPBufs<N>) * (N / 16) * (kTile * 32);
                        const uint32_t d_o = tmem + o_cur + m * N;
                        for (int kk = 0; kk < v16 / 16; ++kk)
                            tc::mma_bf16_elect(d_o, with_addr(dc, cb + kk * 16 * 128),
                                               with_addr(dp, pb + kk * 16 * 32), id_pv,
                                               (first_pv && kk == 0) ? 0u : 1u);
                        release(&bars.pv_empty[s0]);
                        release(&bars.pv_empty[s0 + 1]);
                        rp.advance(CB);
                        rp.advance(CB);
                    }
                    if (!ok) break;
                    tc::commit_elect(smem_u32(&bars.pv_done[t % kPBufs<N>]));
                }
            }
            if (!ok && lane == 0) {
                record_status(a.status, kStatusTimeout);
                ss.abort = 1;
            }
            // drain: every MMA this warp issued has completed before TMEM is freed
            tc::commit_elect(smem_u32(drain));
            if (!__all_sync(0xffffffffu, mbar_wait(smem_u32(drain), 0, lim_ns)) && lane == 0)
                record_status(a.status, kStatusTimeout);
        }
    } else {
        // ================================================================ softmax / epilogue
        griddep_wait();  // before any partial is written (returns at once by the time S arrives)
        SmCtx c;
        c.lane = lane;
        c.tid = tid;
        c.quarter = warp & 3;                 // TMEM lane quarter this warp may access
        c.half = (warp - 4) >> 2;             // which column blocks it owns: half, half+3, ...
        c.tok = c.quarter * 32 + lane;        // token row of the tile
        c.n_own = c.half < N / 16 ? (N / 16 - c.half + 2) / 3 : 0;
        c.group = group;
        c.part = part;
        c.nrc = nrc;
        c.ncc = ncc;
        c.cs = CB;
        c.n_items = n_items;
        c.lane_base = static_cast<uint32_t>(c.quarter * 32) << 16;
        c.tmem = tmem;
        c.o_col0 = o_col0;
        c.ring = ring_b;
        c.p_buf = p_buf;
        c.lim_ns = lim_ns;
        c.t_begin = t_begin;
        c.t_end = t_end;
        softmax_role<N>(c, a, ss, bars);
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, kTmemCols<N>);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

cudaError_t get_encoder()
{
    if (g_encode) return cudaSuccess;
    cudaDriverEntryPointQueryResult q;
    void *fn = nullptr;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return e != cudaSuccess ? e : cudaErrorNotSupported;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return cudaSuccess;
}

// 3-d map over one cache: (columns, tokens per block, blocks), box 64 x box_rows x 1, SW128.
cudaError_t encode_cache_map(CUtensorMap *m, const void *base, int cols, int64_t tok_stride, int64_t blk_stride,
                             int tokens_per_block, int blocks, int box_rows)
{
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(tokens_per_block),
                          static_cast<cuuint64_t>(blocks)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(tok_stride) * 2, static_cast<cuuint64_t>(blk_stride) * 2};
    cuuint32_t box[3] = {64, static_cast<cuuint32_t>(box_rows), 1};
    cuuint32_t es[3] = {1, 1, 1};
    CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <int N, bool SQ>
cudaError_t launch_cfg(const AttnArgs &a, int groups, cudaStream_t st)
{
    cudaError_t e = get_encoder();
    if (e != cudaSuccess) return e;
    const CacheView &c = a.cache;
    const bool paged = c.block_table != nullptr;
    const int tpb = paged ? c.page_size : c.capacity;
    const int blocks = paged ? c.num_pages : a.batch;
    CUtensorMap mc, mr, mq;
    const int box_rows = paged ? kHalf : kTile;
    if ((e = encode_cache_map(&mc, c.c_kv, a.rank, c.c_tok, c.c_blk, tpb, blocks, box_rows)) != cudaSuccess) return e;
    if ((e = encode_cache_map(&mr, c.k_rope, a.d_rope, c.r_tok, c.r_blk, tpb, blocks, box_rows)) != cudaSuccess) return e;
    {
        const int K = a.rank + a.d_rope;
        cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(a.batch) * a.q_len * a.num_heads};
        cuuint64_t strides[1] = {static_cast<cuuint64_t>(K) * 2};
        cuuint32_t box[2] = {64, N};
        cuuint32_t es[2] = {1, 1};
        CUresult r = g_encode(&mq, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(a.q_abs), dims, strides,
                              box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    }
    const int ncc = a.rank / 64;
    const int q_bytes = SQ ? 0 : (((ncc + 1) * N * 128) + 1023) & ~1023;
    const int slot_a = SQ ? kChunkBytes + N * 128 : kChunkBytes;  // QK-ring slot (with its query chunk)
    const int p_bytes = kPBufs<N> * (N / 16) * kTile * 32;
    const int fixed = 1024 /*alignment slack*/ + q_bytes;
    int dev = 0, optin = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    const int static_bytes = static_cast<int>(sizeof(BarsT<N>) + sizeof(Shared<N>) + 32 * 8) + 128;
    const int avail = optin - static_bytes - fixed - p_bytes;
    // the PV ring (refilled from L2) gets six slots where four QK slots still
    // fit beside them (streamed queries), else four or two; the QK ring the
    // rest.  (Measured with 80 rows, whose second P buffer leaves four QK and
    // four PV slots: six PV slots beside three QK slots lose 16 %, two beside
    // five 46 %.)
    int pv_slots = SQ && avail >= 4 * slot_a + 6 * kChunkBytes ? 6 : avail >= 2 * slot_a + 4 * kChunkBytes ? 4 : 2;
    const int cap = tuning().tc_max_slots;  // testing aid: smaller rings
    if (cap >= 4 && pv_slots > cap - 2) pv_slots = 2;
    if (const int v = tuning().tc_pv_slots & ~1; v >= 2 && v <= kMaxSlots && avail >= 2 * slot_a + v * kChunkBytes &&
                                                  (cap < 4 || v <= cap - 2))
        pv_slots = v;  // testing aid
    int qk_slots = (avail - pv_slots * kChunkBytes) / slot_a;
    if (qk_slots > kMaxSlots) qk_slots = kMaxSlots;
    if (cap >= 4 && qk_slots > cap - pv_slots) qk_slots = cap - pv_slots;
    if (qk_slots < 2) return cudaErrorInvalidConfiguration;
    const size_t smem = static_cast<size_t>(fixed) + static_cast<size_t>(qk_slots) * slot_a +
                        static_cast<size_t>(pv_slots) * kChunkBytes + p_bytes;
    if ((e = cudaFuncSetAttribute(attn_tc_kernel<N, SQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(smem))) != cudaSuccess)
        return e;
    TcArgs t;
    t.batch = a.batch;
    t.q_len = a.q_len;
    t.heads = a.num_heads;
    t.rank = a.rank;
    t.d_rope = a.d_rope;
    t.rows = a.q_len * a.num_heads;
    t.num_splits = a.num_splits;
    t.max_kv = a.max_kv;
    t.paged = paged;
    t.bt_stride = c.bt_stride;
    t.num_pages = c.num_pages;
    t.qk_slots = qk_slots;
    t.pv_slots = pv_slots;
    t.scale_log2 = a.sm_scale * 1.4426950408889634f;
    t.kv_len = a.kv_len;
    t.block_table = c.block_table;
    t.o_part = a.o_part;
    t.lse_part = a.lse_part;
    t.o_final = a.o_final;
    t.lse_final = a.lse_final;
    t.status = a.status;
    t.wait_ns = kWaitLimitNs;
    return launch_dependent(attn_tc_kernel<N, SQ>, dim3(groups, a.num_splits, 1), dim3(kThreads), smem, st, 1, t, mc,
                            mr, mq);
}

}  // namespace

TcShape attn_tc_shape(int rows)
{
    // Testing aid: the tuning knob tc_max_rows caps the query rows per CTA (16..80).
    int max_n = tuning().tc_max_rows > 0 ? tuning().tc_max_rows : 80;
    if (max_n < 16) max_n = 16;
    if (max_n > 80) max_n = 80;
    max_n -= max_n % 16;
    TcShape s;
    s.groups = (rows + max_n - 1) / max_n;
    s.n = (((rows + s.groups - 1) / s.groups + 15) / 16) * 16;
    return s;
}

cudaError_t launch_attn_tc(const AttnArgs &a, cudaStream_t st)
{
    const TcShape s = attn_tc_shape(a.q_len * a.num_heads);
    const bool sq = tuning().tc_query != 1;
    switch (s.n) {
    case 16: return sq ? launch_cfg<16, true>(a, s.groups, st) : launch_cfg<16, false>(a, s.groups, st);
    case 32: return sq ? launch_cfg<32, true>(a, s.groups, st) : launch_cfg<32, false>(a, s.groups, st);
    case 48: return sq ? launch_cfg<48, true>(a, s.groups, st) : launch_cfg<48, false>(a, s.groups, st);
    case 64: return sq ? launch_cfg<64, true>(a, s.groups, st) : launch_cfg<64, false>(a, s.groups, st);
    case 80: return sq ? launch_cfg<80, true>(a, s.groups, st) : launch_cfg<80, false>(a, s.groups, st);
    default: return cudaErrorInvalidConfiguration;
    }
}

}  // namespace gbmla

