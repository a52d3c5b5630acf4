// mla_acceptance_stats: acceptance statistics of a draft against its target at
// the same contexts (Sec. 3.3): the overlap alpha_sample = sum_y min(p_D, p_T)
// of the two softmax distributions (Eq. 9) and greedy agreement of their
// argmaxes (Eq. 10), one vocabulary row per context.
//
// Many rows (at least kRowKernelRows): one CTA per row, rows strided over a
// grid of two CTAs per SM.  Pass 1 streams both logit rows from HBM and marks
// their lines evict-last, so that pass 2 reads them again from L2; a CTA moves
// on to its next row as soon as it has written this one, so the SM's loads
// never wait on another CTA's reductions.  Block-wide reductions run in a
// fixed order (bit-reproducible).
//
// Few rows: a row is split over a cluster of kCluster CTAs, each owning a
// contiguous slice of the vocabulary.  When both rows' slices fit in shared memory
// (every vocabulary of the workloads, in bf16), one thread copies them in with
// bulk copies at the start, so the whole slice is in flight at once and HBM is
// read exactly once; both passes then read shared memory.  Otherwise the
// passes stream the slice from global memory (the second from L2).
// Pass 1: maximum, sum of exponentials and first argmax of both rows, a
// vector of 8 (bf16) or 4 (fp32) logits at a time.  The CTAs exchange these
// through distributed shared memory and combine them in rank order (every CTA
// gets the same result, bit for bit).  Pass 2: sum of min(p_D, p_T) over the
// slice; rank 0 adds the slices in rank order.  Exponentials are base 2 with
// log2(e) folded into one FMA, and pass 2 folds the normaliser into the
// exponent, p = 2^(x log2 e - c) with c = m log2 e + log2 Z, so that
// min(p_D, p_T) = 2^min(., .) costs one exponential per token, not two.
#include <math.h>

#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace gbmla {
namespace {

constexpr int kCluster = 8;
constexpr int kAccThreads = 256;
constexpr int kUnroll = 4;                       // streaming path: vectors per tensor per thread in flight
constexpr uint32_t kResidentMax = 200 * 1024;    // shared-memory bytes for both slices
constexpr uint32_t kBulkPiece = 8 * 1024;        // bytes per bulk copy (per row); pass 1 follows the pieces in
constexpr int kMaxPieces = 16;                   // kResidentMax / 2 / kBulkPiece, rounded up

constexpr float kLog2e = 1.4426950408889634f;

struct Stat {
    float m;   // running maximum
    float s;   // sum of exp(x - m) = 2^((x - m) log2 e)
    int idx;   // lowest index holding m
};

// 2^x (the hardware approximation; relative error ~2^-22, and 2^-inf = 0)
__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Sum of f(0) .. f(N-1) as a balanced tree (independent exponentials, a
// dependency chain of log2 N additions rather than N).
template <int N, typename F>
__device__ __forceinline__ float tree_sum(F f)
{
    float v[N];
#pragma unroll
    for (int e = 0; e < N; ++e) v[e] = f(e);
#pragma unroll
    for (int w = 1; w < N; w *= 2)
#pragma unroll
        for (int e = 0; e + w < N; e += 2 * w) v[e] += v[e + w];
    return v[0];
}

// Fold one vector of logits x[0..VN) at indices ybase.. into a: the vector's
// maximum first, so the running base moves (and the sum is rescaled) at most
// once per vector.  A thread visits its indices in increasing order, so an
// equal maximum seen later never displaces the stored index.
template <int VN>
__device__ __forceinline__ void stat_vec(Stat &a, const float (&x)[VN], int ybase)
{
    float vm = x[0];
#pragma unroll
    for (int e = 1; e < VN; ++e) vm = fmaxf(vm, x[e]);
    if (vm > a.m) {
        a.s *= ex2((a.m - vm) * kLog2e);
        a.m = vm;
        int e0 = VN - 1;
#pragma unroll
        for (int e = VN - 1; e >= 0; --e)
            if (x[e] == vm) e0 = e;
        a.idx = ybase + e0;
    }
    const float ml = a.m * kLog2e;
    a.s += tree_sum<VN>([&](int e) { return ex2(fmaf(x[e], kLog2e, -ml)); });
}

__device__ __forceinline__ void stat_one(Stat &a, float x, int y)
{
    const float v[1] = {x};
    stat_vec<1>(a, v, y);
}

__device__ __forceinline__ Stat stat_merge(Stat a, Stat b)
{
    if (b.s == 0.f) return a;
    if (a.s == 0.f) return b;
    if (b.m > a.m || (b.m == a.m && b.idx < a.idx)) {
        const Stat t = a;
        a = b;
        b = t;
    }
    a.s += b.s * ex2((b.m - a.m) * kLog2e);  // a.m >= b.m
    return a;
}

// ---- packed forms for bf16 logits (fewer instructions per token): the
// vector maximum on raw bf16 pairs (exact), the exponent arguments and the
// sums of exponentials as two-wide fp32 FMAs and adds (each lane rounds as
// the scalar instruction does).
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b)
{
    uint32_t r;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

__device__ __forceinline__ uint64_t pk(float lo, float hi)
{
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}

__device__ __forceinline__ void upk(uint64_t v, float &lo, float &hi)
{
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}

__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c)
{
    uint64_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}

__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b)
{
    uint64_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}

// both logits of a bf16 pair as a packed fp32 pair (element 2k in the low half)
__device__ __forceinline__ uint64_t bf16x2_f32x2(uint32_t w) { return pk(bf16_lo(w), bf16_hi(w)); }

// Sum of 2^(t_e) over the four packed pairs t[0..3] (a tree of packed adds).
__device__ __forceinline__ float ex2_sum8(const uint64_t (&t)[4])
{
    uint64_t e[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        float a, b;
        upk(t[q], a, b);
        e[q] = pk(ex2(a), ex2(b));
    }
    const uint64_t s = add2(add2(e[0], e[1]), add2(e[2], e[3]));
    float lo, hi;
    upk(s, lo, hi);
    return lo + hi;
}

// stat_vec for eight bf16 logits in their raw 16-byte vector.
__device__ __forceinline__ void stat_bf16(Stat &a, const uint4 &v, int ybase)
{
    const uint32_t mw = bmax2(bmax2(v.x, v.y), bmax2(v.z, v.w));
    const float vm = fmaxf(bf16_lo(mw), bf16_hi(mw));
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    if (vm > a.m) {
        a.s *= ex2((a.m - vm) * kLog2e);
        a.m = vm;
        int e0 = 7;
#pragma unroll
        for (int e = 7; e >= 0; --e)
            if (((e & 1) ? bf16_hi(w[e >> 1]) : bf16_lo(w[e >> 1])) == vm) e0 = e;
        a.idx = ybase + e0;
    }
    const float nml = -(a.m * kLog2e);
    const uint64_t L = pk(kLog2e, kLog2e), C = pk(nml, nml);
    uint64_t t[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) t[q] = fma2(bf16x2_f32x2(w[q]), L, C);
    a.s += ex2_sum8(t);
}

// Sum over eight bf16 token pairs of min(p_D, p_T) = 2^min(x_D log2 e - c_D, x_T log2 e - c_T).
__device__ __forceinline__ float pmin_bf16(const uint4 &vd, const uint4 &vt, float cd, float ct)
{
    const uint64_t L = pk(kLog2e, kLog2e), CD = pk(-cd, -cd), CT = pk(-ct, -ct);
    const uint32_t wd[4] = {vd.x, vd.y, vd.z, vd.w}, wt[4] = {vt.x, vt.y, vt.z, vt.w};
    uint64_t t[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        float d0, d1, t0, t1;
        upk(fma2(bf16x2_f32x2(wd[q]), L, CD), d0, d1);
        upk(fma2(bf16x2_f32x2(wt[q]), L, CT), t0, t1);
        t[q] = pk(fminf(d0, t0), fminf(d1, t1));
    }
    return ex2_sum8(t);
}

template <typename T>
struct Vec;
template <>
struct Vec<float> {
    static constexpr int n = 4;
    __device__ static void load(const float *p, float (&x)[4], bool stream)
    {
        const float4 v = stream ? __ldcs(reinterpret_cast<const float4 *>(p)) : *reinterpret_cast<const float4 *>(p);
        x[0] = v.x;
        x[1] = v.y;
        x[2] = v.z;
        x[3] = v.w;
    }
    __device__ static void cvt(const uint4 &w, float (&x)[4])
    {
        x[0] = __uint_as_float(w.x);
        x[1] = __uint_as_float(w.y);
        x[2] = __uint_as_float(w.z);
        x[3] = __uint_as_float(w.w);
    }
    __device__ static float one(const float *p) { return *p; }
};
template <>
struct Vec<uint16_t> {
    static constexpr int n = 8;
    __device__ static void load(const uint16_t *p, float (&x)[8], bool stream)
    {
        const uint4 v = stream ? __ldcs(reinterpret_cast<const uint4 *>(p)) : *reinterpret_cast<const uint4 *>(p);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            x[2 * e] = __uint_as_float(w[e] << 16);
            x[2 * e + 1] = __uint_as_float(w[e] & 0xffff0000u);
        }
    }
    __device__ static void cvt(const uint4 &v, float (&x)[8])
    {
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            x[2 * e] = __uint_as_float(w[e] << 16);
            x[2 * e + 1] = __uint_as_float(w[e] & 0xffff0000u);
        }
    }
    __device__ static float one(const uint16_t *p) { return __uint_as_float(static_cast<uint32_t>(*p) << 16); }
};

// 16 bytes from global memory with an L2 eviction policy.
__device__ __forceinline__ uint4 ld_hint16(const void *p, uint64_t pol)
{
    uint4 w;
    asm volatile("ld.global.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=r"(w.x), "=r"(w.y), "=r"(w.z), "=r"(w.w)
                 : "l"(p), "l"(pol));
    return w;
}

// Reduction over the 32 lanes of a warp by shuffles; every lane gets the result.
template <typename V, typename Op>
__device__ __forceinline__ V warp_reduce(V v, Op op)
{
    for (int o = 16; o > 0; o >>= 1) {
        V w;
        if constexpr (sizeof(V) == sizeof(float)) {
            w = __shfl_xor_sync(0xffffffffu, v, o);
        } else {
            w.m = __shfl_xor_sync(0xffffffffu, v.m, o);
            w.s = __shfl_xor_sync(0xffffffffu, v.s, o);
            w.idx = __shfl_xor_sync(0xffffffffu, v.idx, o);
        }
        v = op(v, w);
    }
    return v;
}

// Block-wide reduction of a value with `op` (identity `id`); every thread gets
// the result.  Each warp reduces by shuffles, then warp 0 reduces the warps'
// partials the same way and publishes the result (a fixed tree: the bits do
// not depend on timing).  `scratch` holds NT / 32 + 1 values.
template <int NT = kAccThreads, typename V, typename Op>
__device__ V block_reduce(V v, Op op, V *scratch, V id)
{
    v = warp_reduce(v, op);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();  // (the previous reduction's result has been read)
    if (lane == 0) scratch[warp] = v;
    __syncthreads();
    if (warp == 0) {
        V r = warp_reduce(lane < NT / 32 ? scratch[lane] : id, op);
        if (lane == 0) scratch[NT / 32] = r;
    }
    __syncthreads();
    return scratch[NT / 32];
}

__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t mbar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(mbar)
                 : "memory");
}

// RESIDENT: the slice is copied into shared memory first (and read there).
template <typename T, bool RESIDENT>
__global__ void __launch_bounds__(kAccThreads) accept_kernel(int vocab, int64_t stride, int chunk,
                                                            const T *__restrict__ draft,
                                                            const T *__restrict__ target, float *alpha,
                                                            int32_t *argmax_d, int32_t *argmax_t, int32_t *greedy,
                                                            unsigned *status)
{
    extern __shared__ __align__(16) unsigned char acc_smem[];
    __shared__ Stat s_stat[kCluster][2];        // (draft, target) statistics of every rank, pushed here by each
    __shared__ float s_part[kCluster];          // every rank's share of the overlap (rank 0's copy is read)
    __shared__ Stat scratch_s[kAccThreads / 32 + 1];
    __shared__ float scratch_f[kAccThreads / 32 + 1];
    __shared__ __align__(8) uint64_t bar[kMaxPieces];
    constexpr int VN = Vec<T>::n;
    const int rank = blockIdx.x % kCluster;
    const int64_t row = blockIdx.y;
    const int y0 = rank * chunk, y1 = min(vocab, y0 + chunk);  // chunk is a multiple of VN
    const int n = y1 > y0 ? y1 - y0 : 0;
    const int nvec = n / VN;                                    // whole vectors; then the row's tail
    const T *gd_row = draft + row * stride + y0, *gt_row = target + row * stride + y0;
    const T *d = gd_row, *t = gt_row;                           // where the passes read the slice
    bool landed = true;                                         // the bulk copies have arrived
    // the cluster's CTAs must all have started before one writes another's
    // shared memory: arrive now, wait just before the first such write
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    // resident: piece k = bytes [k kBulkPiece, (k + 1) kBulkPiece) of both rows, landing on bar[k]
    const uint32_t bytes = RESIDENT ? static_cast<uint32_t>(nvec) * VN * sizeof(T) : 0u;  // a multiple of 16
    const int pieces = static_cast<int>((bytes + kBulkPiece - 1) / kBulkPiece);
    if (RESIDENT) {
        const uint32_t pad = (static_cast<uint32_t>(chunk) * sizeof(T) + 15u) & ~15u;
        const T *sd_buf = reinterpret_cast<const T *>(acc_smem), *st_buf = reinterpret_cast<const T *>(acc_smem + pad);
        if (threadIdx.x == 0) {
            for (int k = 0; k < pieces; ++k) mbar_init(&bar[k], 1);
            tc::fence_barrier_init();
        }
        __syncthreads();
        griddep_wait();
        griddep_launch_dependents();
        if (threadIdx.x == 0) {
            for (int k = 0; k < pieces; ++k) {
                const uint32_t o = k * kBulkPiece, len = bytes - o < kBulkPiece ? bytes - o : kBulkPiece;
                const uint32_t b = smem_u32(&bar[k]);
                tc::mbar_arrive_expect_tx(b, 2 * len);
                bulk_load(smem_u32(sd_buf) + o, reinterpret_cast<const unsigned char *>(gd_row) + o, len, b);
                bulk_load(smem_u32(st_buf) + o, reinterpret_cast<const unsigned char *>(gt_row) + o, len, b);
            }
        }
        d = sd_buf;
        t = st_buf;
    } else {
        griddep_wait();
        griddep_launch_dependents();
    }

    // ---- pass 1: maxima, sums, argmaxes
    Stat sd{-INFINITY, 0.f, 0x7fffffff}, st{-INFINITY, 0.f, 0x7fffffff};
    if (RESIDENT) {
        constexpr int kPieceVecs = kBulkPiece / 16;  // 16-byte vectors per piece and row
        for (int k = 0; k < pieces; ++k) {
            // a wait that runs out is recorded, and the piece is read from global memory instead
            const bool ok = __syncthreads_and(mbar_wait(smem_u32(&bar[k]), 0, kWaitLimitNs));
            if (!ok) {
                landed = false;
                if (threadIdx.x == 0) record_status(status, kStatusTimeout);
            }
            const T *pd = ok ? d : gd_row, *pt = ok ? t : gt_row;
            const int v1 = min(nvec, (k + 1) * kPieceVecs);
            for (int v = k * kPieceVecs + threadIdx.x; v < v1; v += kAccThreads) {
                float xd[VN], xt[VN];
                Vec<T>::load(pd + v * VN, xd, false);
                Vec<T>::load(pt + v * VN, xt, false);
                stat_vec<VN>(sd, xd, y0 + v * VN);
                stat_vec<VN>(st, xt, y0 + v * VN);
            }
        }
        if (!landed) {  // pass 2 reads global memory
            d = gd_row;
            t = gt_row;
        }
    } else {
        for (int v0 = threadIdx.x; v0 < nvec; v0 += kAccThreads * kUnroll) {
            float xd[kUnroll][VN], xt[kUnroll][VN];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int v = v0 + u * kAccThreads;
                if (v < nvec) {
                    Vec<T>::load(d + v * VN, xd[u], false);
                    Vec<T>::load(t + v * VN, xt[u], false);
                }
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int v = v0 + u * kAccThreads;
                if (v < nvec) {
                    stat_vec<VN>(sd, xd[u], y0 + v * VN);
                    stat_vec<VN>(st, xt[u], y0 + v * VN);
                }
            }
        }
    }
    for (int i = nvec * VN + threadIdx.x; i < n; i += kAccThreads) {  // the row's tail, from global memory
        stat_one(sd, Vec<T>::one(gd_row + i), y0 + i);
        stat_one(st, Vec<T>::one(gt_row + i), y0 + i);
    }
    auto merge = [](Stat a, Stat b) { return stat_merge(a, b); };
    const Stat none{-INFINITY, 0.f, 0x7fffffff};
    sd = block_reduce(sd, merge, scratch_s, none);
    st = block_reduce(st, merge, scratch_s, none);
    // push this rank's statistics into slot [rank] of every rank, then combine
    // all slots in rank order (every CTA computes the same bits)
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
    if (threadIdx.x < kCluster) {
        const uint32_t local = smem_u32(&s_stat[rank][0]);
        uint32_t remote;
        asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(static_cast<int>(threadIdx.x)));
        // scalar stores: a Stat is 12 bytes, only 4-byte aligned
        asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote), "f"(sd.m) : "memory");
        asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote + 4), "f"(sd.s) : "memory");
        asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(remote + 8), "r"(sd.idx) : "memory");
        asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote + 12), "f"(st.m) : "memory");
        asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote + 16), "f"(st.s) : "memory");
        asm volatile("st.shared::cluster.s32 [%0], %1;" ::"r"(remote + 20), "r"(st.idx) : "memory");
    }
    tc::cluster_sync();
    Stat gd{-INFINITY, 0.f, 0x7fffffff}, gt{-INFINITY, 0.f, 0x7fffffff};
    for (int r = 0; r < kCluster; ++r) {
        gd = stat_merge(gd, s_stat[r][0]);
        gt = stat_merge(gt, s_stat[r][1]);
    }
    // p = exp(x - m) / Z = 2^(x log2 e - c), c = m log2 e + log2 Z
    const float cd = gd.m * kLog2e + log2f(gd.s), ct = gt.m * kLog2e + log2f(gt.s);
    auto pmin = [&](float xd, float xt) { return ex2(fminf(fmaf(xd, kLog2e, -cd), fmaf(xt, kLog2e, -ct))); };

    // ---- pass 2: sum of min(p_D, p_T) over the slice
    float acc = 0.f;
    if (RESIDENT) {
        float acc2 = 0.f;  // two vectors per step, two accumulators
        for (int v = threadIdx.x; v < nvec; v += 2 * kAccThreads) {
            float xd[VN], xt[VN], yd[VN], yt[VN];
            const bool second = v + kAccThreads < nvec;
            Vec<T>::load(d + v * VN, xd, false);
            Vec<T>::load(t + v * VN, xt, false);
            if (second) {
                Vec<T>::load(d + (v + kAccThreads) * VN, yd, false);
                Vec<T>::load(t + (v + kAccThreads) * VN, yt, false);
            }
            acc += tree_sum<VN>([&](int e) { return pmin(xd[e], xt[e]); });
            if (second) acc2 += tree_sum<VN>([&](int e) { return pmin(yd[e], yt[e]); });
        }
        acc += acc2;
    } else {
        for (int v0 = threadIdx.x; v0 < nvec; v0 += kAccThreads * kUnroll) {
            float xd[kUnroll][VN], xt[kUnroll][VN];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int v = v0 + u * kAccThreads;
                if (v < nvec) {
                    Vec<T>::load(d + v * VN, xd[u], true);
                    Vec<T>::load(t + v * VN, xt[u], true);
                }
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int v = v0 + u * kAccThreads;
                if (v < nvec) {
#pragma unroll
                    for (int e = 0; e < VN; ++e) acc += pmin(xd[u][e], xt[u][e]);
                }
            }
        }
    }
    for (int i = nvec * VN + threadIdx.x; i < n; i += kAccThreads)
        acc += pmin(Vec<T>::one(gd_row + i), Vec<T>::one(gt_row + i));
    acc = block_reduce(acc, [](float a, float b) { return a + b; }, scratch_f, 0.f);
    if (threadIdx.x == 0) {  // this rank's share into slot [rank] of rank 0
        uint32_t remote;
        asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(&s_part[rank])), "r"(0));
        asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote), "f"(acc) : "memory");
    }
    tc::cluster_sync();
    if (rank == 0 && threadIdx.x == 0) {
        float total = 0.f;
        for (int r = 0; r < kCluster; ++r) total += s_part[r];  // rank order
        if (alpha) alpha[row] = total;
        if (argmax_d) argmax_d[row] = gd.idx;
        if (argmax_t) argmax_t[row] = gt.idx;
        if (greedy) greedy[row] = gd.idx == gt.idx;
    }
    if (RESIDENT && !landed)  // pieces still in flight land before the CTA leaves
        for (int k = 0; k < pieces; ++k) mbar_wait(smem_u32(&bar[k]), 0, kWaitLimitNs);
}

// ---------------------------------------------------------------- one CTA per row

constexpr int kRowThreads = 512;
constexpr int kRowUnroll = 2;      // vectors per tensor per thread in flight
constexpr int kRowKernelRows = 128;

template <typename T>
__global__ void __launch_bounds__(kRowThreads, 2) accept_row_kernel(int rows, int vocab, int64_t stride,
                                                                const T *__restrict__ draft,
                                                                const T *__restrict__ target, float *alpha,
                                                                int32_t *argmax_d, int32_t *argmax_t,
                                                                int32_t *greedy)
{
    __shared__ Stat scratch_s[kRowThreads / 32 + 1];
    __shared__ float scratch_f[kRowThreads / 32 + 1];
    griddep_wait();
    griddep_launch_dependents();
    constexpr int VN = Vec<T>::n;
    const int nvec = vocab / VN;
    const uint64_t keep = tc::policy_evict_last(), drop = tc::policy_evict_first();
    auto merge = [](Stat a, Stat b) { return stat_merge(a, b); };
    for (int64_t row = blockIdx.x; row < rows; row += gridDim.x) {
        const T *d = draft + row * stride, *t = target + row * stride;
        // ---- pass 1: maxima, sums, argmaxes (lines kept in L2 for pass 2)
        Stat sd{-INFINITY, 0.f, 0x7fffffff}, st{-INFINITY, 0.f, 0x7fffffff};
        for (int v0 = threadIdx.x; v0 < nvec; v0 += kRowThreads * kRowUnroll) {
            uint4 wd[kRowUnroll], wt[kRowUnroll];
#pragma unroll
            for (int u = 0; u < kRowUnroll; ++u) {
                const int v = v0 + u * kRowThreads;
                if (v < nvec) {
                    wd[u] = ld_hint16(d + static_cast<int64_t>(v) * VN, keep);
                    wt[u] = ld_hint16(t + static_cast<int64_t>(v) * VN, keep);
                }
            }
#pragma unroll
            for (int u = 0; u < kRowUnroll; ++u) {
                const int v = v0 + u * kRowThreads;
                if (v < nvec) {
                    if constexpr (sizeof(T) == 2) {
                        stat_bf16(sd, wd[u], v * VN);
                        stat_bf16(st, wt[u], v * VN);
                    } else {
                        float xd[VN], xt[VN];
                        Vec<T>::cvt(wd[u], xd);
                        Vec<T>::cvt(wt[u], xt);
                        stat_vec<VN>(sd, xd, v * VN);
                        stat_vec<VN>(st, xt, v * VN);
                    }
                }
            }
        }
        for (int i = nvec * VN + threadIdx.x; i < vocab; i += kRowThreads) {  // the row's tail
            stat_one(sd, Vec<T>::one(d + i), i);
            stat_one(st, Vec<T>::one(t + i), i);
        }
        const Stat none{-INFINITY, 0.f, 0x7fffffff};
        sd = block_reduce<kRowThreads>(sd, merge, scratch_s, none);
        st = block_reduce<kRowThreads>(st, merge, scratch_s, none);
        const float cd = sd.m * kLog2e + log2f(sd.s), ct = st.m * kLog2e + log2f(st.s);
        auto pmin = [&](float xd, float xt) { return ex2(fminf(fmaf(xd, kLog2e, -cd), fmaf(xt, kLog2e, -ct))); };
        // ---- pass 2: sum of min(p_D, p_T), a last read of the lines
        float acc = 0.f, acc2 = 0.f;
        for (int v0 = threadIdx.x; v0 < nvec; v0 += kRowThreads * kRowUnroll) {
            uint4 wd[kRowUnroll], wt[kRowUnroll];
#pragma unroll
            for (int u = 0; u < kRowUnroll; ++u) {
                const int v = v0 + u * kRowThreads;
                if (v < nvec) {
                    wd[u] = ld_hint16(d + static_cast<int64_t>(v) * VN, drop);
                    wt[u] = ld_hint16(t + static_cast<int64_t>(v) * VN, drop);
                }
            }
#pragma unroll
            for (int u = 0; u < kRowUnroll; ++u) {
                const int v = v0 + u * kRowThreads;
                if (v < nvec) {
                    float a;
                    if constexpr (sizeof(T) == 2) {
                        a = pmin_bf16(wd[u], wt[u], cd, ct);
                    } else {
                        float xd[VN], xt[VN];
                        Vec<T>::cvt(wd[u], xd);
                        Vec<T>::cvt(wt[u], xt);
                        a = tree_sum<VN>([&](int e) { return pmin(xd[e], xt[e]); });
                    }
                    if (u & 1)
                        acc2 += a;
                    else
                        acc += a;
                }
            }
        }
        acc += acc2;
        for (int i = nvec * VN + threadIdx.x; i < vocab; i += kRowThreads)
            acc += pmin(Vec<T>::one(d + i), Vec<T>::one(t + i));
        acc = block_reduce<kRowThreads>(acc, [](float a, float b) { return a + b; }, scratch_f, 0.f);
        if (threadIdx.x == 0) {
            if (alpha) alpha[row] = acc;
            if (argmax_d) argmax_d[row] = sd.idx;
            if (argmax_t) argmax_t[row] = st.idx;
            if (greedy) greedy[row] = sd.idx == st.idx;
        }
    }
}

template <typename T>
cudaError_t launch_typed(int rows, int vocab, const void *draft, const void *target, int64_t stride, float *alpha,
                         int32_t *argmax_d, int32_t *argmax_t, int32_t *greedy, unsigned *status, cudaStream_t st)
{
    constexpr int vn = Vec<T>::n;
    if (rows >= kRowKernelRows) {
        int dev = 0, sms = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        const int grid = rows < 2 * sms ? rows : 2 * sms;
        return launch_dependent(accept_row_kernel<T>, dim3(grid), dim3(kRowThreads), 0, st, 1, rows, vocab, stride,
                                static_cast<const T *>(draft), static_cast<const T *>(target), alpha, argmax_d,
                                argmax_t, greedy);
    }
    int chunk = (vocab + kCluster - 1) / kCluster;
    chunk = (chunk + vn - 1) / vn * vn;
    const uint32_t pad = (static_cast<uint32_t>(chunk) * sizeof(T) + 15u) & ~15u;
    const dim3 grid(kCluster, rows);
    const T *dp = static_cast<const T *>(draft), *tp = static_cast<const T *>(target);
    if (2 * pad <= kResidentMax) {
        cudaError_t e = cudaFuncSetAttribute(accept_kernel<T, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(2 * pad));
        if (e != cudaSuccess) return e;
        return launch_dependent(accept_kernel<T, true>, grid, dim3(kAccThreads), 2 * pad, st, kCluster, vocab, stride,
                                chunk, dp, tp, alpha, argmax_d, argmax_t, greedy, status);
    }
    return launch_dependent(accept_kernel<T, false>, grid, dim3(kAccThreads), 0, st, kCluster, vocab, stride, chunk,
                            dp, tp, alpha, argmax_d, argmax_t, greedy, status);
}

}  // namespace

cudaError_t launch_acceptance(int rows, int vocab, int dtype, const void *draft, const void *target, int64_t stride,
                              float *alpha, int32_t *argmax_d, int32_t *argmax_t, int32_t *greedy, unsigned *status,
                              cudaStream_t st)
{
    if (rows <= 0) return cudaSuccess;
    if (dtype == 0)
        return launch_typed<float>(rows, vocab, draft, target, stride, alpha, argmax_d, argmax_t, greedy, status, st);
    return launch_typed<uint16_t>(rows, vocab, draft, target, stride, alpha, argmax_d, argmax_t, greedy, status, st);
}

}  // namespace gbmla
