// Device-side helpers shared by the kernels of libgbmla.so.
#pragma once

#include <math.h>

#include <utility>

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/gbmla.h"

namespace gbmla {

// Bits of the sticky per-device status word (read by mla_check_status).
enum : unsigned { kStatusBounds = 1u, kStatusTimeout = 2u };

// Default limit of every bounded device-side wait (about a second).
constexpr uint64_t kWaitLimitNs = 1000000000ull;

__device__ __forceinline__ void record_status(unsigned *status, unsigned bits)
{
    atomicOr(status, bits);
}

__device__ __forceinline__ uint64_t global_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ float bf16_bits_to_float(uint16_t b)
{
    return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ---------------------------------------------------------------- mbarriers

__device__ __forceinline__ void mbar_init(uint64_t *bar, unsigned count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait until the phase with the given parity of the mbarrier at shared
// address `bar` has completed, for at most `limit_ns` nanoseconds.  Returns
// false if the limit ran out (the caller records a timeout and winds down).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns)
{
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (;;) {
        for (int i = 0; i < 32; ++i)
            if (mbar_try_wait(bar, parity)) return true;
        if (global_ns() - t0 > limit_ns) return false;
    }
}

// ---------------------------------------------------------------- dependent launch
// The kernels of a decode step are launched as programmatic dependents of
// the previous launch: a kernel's prologue (barrier set-up, TMEM allocation,
// descriptor prefetch) may run while its predecessor drains, and
// griddep_wait() returns once the predecessor has completed with its memory
// visible.  Both are no-ops for a kernel launched without the attribute.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents()
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launch `kernel` on `st` as a programmatic dependent of the stream's
// previous work (plus an optional cluster size).
template <typename... KArgs, typename... Args>
cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                             int cluster, Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    int n = 0;
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
    if (cluster > 1) {
        attr[n].id = cudaLaunchAttributeClusterDimension;
        attr[n].val.clusterDim.x = cluster;
        attr[n].val.clusterDim.y = 1;
        attr[n].val.clusterDim.z = 1;
        ++n;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ---------------------------------------------------------------- split-KV partition
// Tiles of MLA_SPLIT_TILE tokens of all sequences, in batch order, form one
// list of T tiles; partition k owns tiles [floor(k*T/S), floor((k+1)*T/S)).

__device__ __forceinline__ int64_t part_begin(int64_t k, int64_t T, int S)
{
    return (k * T) / S;
}

// Largest k whose range starts at or before tile t (the non-empty partition
// holding tile t).
__device__ __forceinline__ int part_of_tile(int64_t t, int64_t T, int S)
{
    return static_cast<int>(((t + 1) * S - 1) / T);
}

// Tiles of a sequence with kv cached tokens; a length the kernels cannot
// serve (kv < q_len or kv > capacity) counts as zero tiles everywhere, so
// every kernel derives the same partition from the same kv_len.
__device__ __forceinline__ int64_t seq_tiles(int kv, int q_len, int capacity)
{
    if (kv < q_len || kv > capacity || kv <= 0) return 0;
    return (kv + MLA_SPLIT_TILE - 1) / MLA_SPLIT_TILE;
}

// Block-wide sum of seq_tiles over sequences [0, n); every thread gets it.
// Uses `red` (>= 32 int64) of shared scratch.  All threads must call it.
// `groups` > 1: unit b of n is group b % groups of sequence b / groups (its
// length is kv_len[b / groups]).
__device__ __forceinline__ int64_t block_tile_sum(const int32_t *kv_len, int n, int q_len, int capacity,
                                                  int64_t *red, int groups = 1)
{
    int64_t acc = 0;
    for (int b = threadIdx.x; b < n; b += blockDim.x) acc += seq_tiles(kv_len[b / groups], q_len, capacity);
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) red[warp] = acc;
    __syncthreads();
    int64_t tot = 0;
    const int nw = (blockDim.x + 31) >> 5;
    for (int w = 0; w < nw; ++w) tot += red[w];
    __syncthreads();
    return tot;
}

// One pass over the lengths: *total = all sequences' tiles, *before = the
// tiles of sequences 0 .. b-1 (block-wide; every thread gets both).
__device__ __forceinline__ void block_tile_sums(const int32_t *kv_len, int n, int b, int q_len, int capacity,
                                                int64_t *red, int64_t *total, int64_t *before, int groups = 1)
{
    int64_t acc = 0, pre = 0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const int64_t t = seq_tiles(kv_len[i / groups], q_len, capacity);
        acc += t;
        if (i < b) pre += t;
    }
    for (int o = 16; o > 0; o >>= 1) {
        acc += __shfl_xor_sync(0xffffffffu, acc, o);
        pre += __shfl_xor_sync(0xffffffffu, pre, o);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __syncthreads();
    if (lane == 0) {
        red[2 * warp] = acc;
        red[2 * warp + 1] = pre;
    }
    __syncthreads();
    int64_t tot = 0, bef = 0;
    const int nw = (blockDim.x + 31) >> 5;
    for (int w = 0; w < nw; ++w) {
        tot += red[2 * w];
        bef += red[2 * w + 1];
    }
    __syncthreads();
    *total = tot;
    *before = bef;
}


// RoPE frequencies (Sec. 3.1, theta_k = base^(-2k/d_rope)) as fixed-point
// fractions of a turn, f_k = round(theta_k / (2 pi) * 2^64), computed once on
// the host.  The angle of position pos is then pos * f_k mod 2^64 turns: one
// exact integer multiply does the range reduction for any position, and the
// result, read as a signed fraction x in [-1, 1), is the angle pi * x that
// sincospif evaluates in fp32.  No fp64 arithmetic runs on the device.
struct RopeTurns {
    uint64_t f[64];  // d / 2 <= 64 frequencies (positional keys of MLA, whole GQA heads up to 128)
};

inline RopeTurns rope_turns(int d_rope, float base)
{
    RopeTurns t{};
    const double two_pi = 6.283185307179586476925286766559;
    for (int k = 0; k < d_rope / 2 && k < 64; ++k) {
        const double theta = pow(static_cast<double>(base), -2.0 * k / d_rope);  // <= 1
        t.f[k] = static_cast<uint64_t>(ldexp(theta / two_pi, 64));                // < 2^62
    }
    return t;
}

__device__ __forceinline__ void rope_cos_sin(int64_t pos, uint64_t f, float *c, float *s)
{
    const uint64_t turn = static_cast<uint64_t>(pos) * f;                                   // mod 2^64
    const float x = static_cast<float>(static_cast<int64_t>(turn)) * 1.0842021724855044e-19f;  // 2^-63
    sincospif(x, s, c);
}

}  // namespace gbmla
