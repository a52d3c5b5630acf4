// The projections of the decode step as grouped GEMMs (all bf16 weights,
// fp32 accumulation, bf16 results):
//   absorption (Sec. 1; Eq. 5 read right to left): q_lat[row] = q_nope[row] W_UK[g]   (W_UK: d_nope x r)
//   value up-projection (Eq. 5):                    o[row]     = W_UV[g] o_lat[row]    (W_UV: d_v x r)
//   output projection (Sec. 4.1):                   out[m]     = W_O concat_h o[m]     (W_O: D x H d_v)
// In every case C[phys(g, m), n] = sum_k A[phys(g, m), k] B_g(n, k) for the M
// rows of group g, with phys(g, m) = (m / hpg) * blk + g * hpg + m % hpg.
//
// Up to 32 rows and a deep K (the output projection of a small batch): a
// CUDA-core kernel that streams each weight once (the product is weight-
// bandwidth bound).  Otherwise: a tcgen05 GEMM,
// 128 rows x BN columns per CTA, the A rows gathered (and converted from fp32
// where the source is fp32) by four warps into 128B-swizzled K-major tiles,
// the weight tile loaded by TMA, the accumulator in TMEM.
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

__device__ __forceinline__ float a_value(const GroupGemm &p, int64_t row, int k)
{
    return p.a_f32 ? static_cast<const float *>(p.A)[row * p.lda + k]
                   : bf16_bits_to_float(static_cast<const uint16_t *>(p.A)[row * p.lda + k]);
}

__device__ __forceinline__ void store_bf16(const GroupGemm &p, int64_t row, int n, float v)
{
    static_cast<uint16_t *>(p.C)[row * p.ldc + n] = __bfloat16_as_ushort(__float2bfloat16_rn(v));
}

// ---------------------------------------------------------------- few rows, K-major weights
// B_g(n, k) = B[g N K + n K + k].  The group's A rows sit in shared memory
// as fp32 [M][K]; a warp owns 2 columns n, each lane walks K in 8-element
// (16-byte) steps, four steps in flight, so every weight row is read once,
// coalesced, with enough bytes in flight to stream at memory speed.
constexpr int kSmallWarps = 8;
constexpr int kSmallCols = 2 * kSmallWarps;  // columns per block

__global__ void __launch_bounds__(32 * kSmallWarps) small_kmajor_kernel(GroupGemm p)
{
    extern __shared__ float As[];
    const int g = blockIdx.y;
    // stage A (K is a multiple of 8: 8-element vectors)
    const int kv = p.K / 8;
    for (int i = threadIdx.x; i < p.M * kv; i += blockDim.x) {
        const int m = i / kv, k = (i - m * kv) * 8;
        const int64_t row = phys_row(p, g, m);
        float v[8];
        if (p.a_f32) {
            const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(p.A) + row * p.lda + k);
            const float4 x = src[0], y = src[1];
            v[0] = x.x, v[1] = x.y, v[2] = x.z, v[3] = x.w, v[4] = y.x, v[5] = y.y, v[6] = y.z, v[7] = y.w;
        } else {
            const uint4 w = *reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(p.A) + row * p.lda + k);
            const uint32_t u[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                v[2 * e] = __uint_as_float(u[e] << 16);
                v[2 * e + 1] = __uint_as_float(u[e] & 0xffff0000u);
            }
        }
        float4 *dst = reinterpret_cast<float4 *>(As + m * p.K + k);
        dst[0] = make_float4(v[0], v[1], v[2], v[3]);
        dst[1] = make_float4(v[4], v[5], v[6], v[7]);
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n0 = blockIdx.x * kSmallCols + warp * 2;
    const uint16_t *B = static_cast<const uint16_t *>(p.B) + static_cast<int64_t>(g) * p.N * p.K;
    for (int m0 = 0; m0 < p.M; m0 += 8) {
        float acc[2][8];
#pragma unroll
        for (int f = 0; f < 2; ++f)
#pragma unroll
            for (int r = 0; r < 8; ++r) acc[f][r] = 0.f;
        for (int kb = 8 * lane; kb < p.K; kb += 4 * 256) {
            uint4 w[4][2];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int f = 0; f < 2; ++f) {
                    const int k0 = kb + 256 * u;
                    w[u][f] = (k0 < p.K && n0 + f < p.N)
                                  ? *reinterpret_cast<const uint4 *>(B + static_cast<int64_t>(n0 + f) * p.K + k0)
                                  : make_uint4(0, 0, 0, 0);
                }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int k0 = kb + 256 * u;
                if (k0 >= p.K) break;
                float wf[2][8];
#pragma unroll
                for (int f = 0; f < 2; ++f) {
                    const uint32_t uu[4] = {w[u][f].x, w[u][f].y, w[u][f].z, w[u][f].w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        wf[f][2 * e] = __uint_as_float(uu[e] << 16);
                        wf[f][2 * e + 1] = __uint_as_float(uu[e] & 0xffff0000u);
                    }
                }
#pragma unroll
                for (int r = 0; r < 8; ++r) {
                    if (m0 + r < p.M) {
                        const float4 a0 = *reinterpret_cast<const float4 *>(As + (m0 + r) * p.K + k0);
                        const float4 a1 = *reinterpret_cast<const float4 *>(As + (m0 + r) * p.K + k0 + 4);
                        const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
#pragma unroll
                        for (int f = 0; f < 2; ++f)
#pragma unroll
                            for (int e = 0; e < 8; ++e) acc[f][r] = fmaf(wf[f][e], av[e], acc[f][r]);
                    }
                }
            }
        }
#pragma unroll
        for (int f = 0; f < 2; ++f)
#pragma unroll
            for (int r = 0; r < 8; ++r) {
                float v = acc[f][r];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                if (lane == f * 8 + r && n0 + f < p.N && m0 + r < p.M) store_bf16(p, phys_row(p, g, m0 + r), n0 + f, v);
            }
    }
}

// ---------------------------------------------------------------- tensor-core GEMM
constexpr int kStages = 4;
constexpr int kTileM = 128;
constexpr int kGemmThreads = 192;  // warp 0 TMA, warp 1 MMA, warps 2..5 A rows / epilogue

struct __align__(8) GemmBars {
    uint64_t full_a[kStages], full_b[kStages], empty[kStages], done;
};

// BN: columns per CTA (64, 128 or 256).  NMAJ: the weight is N-major.
template <int BN, bool NMAJ>
__global__ void __launch_bounds__(kGemmThreads) gemm_tc_kernel(const __grid_constant__ GroupGemm p,
                                                               const __grid_constant__ CUtensorMap map_b)
{
    constexpr int kABytes = kTileM * 128;  // 128 rows x 64 K, bf16, SW128 K-major
    constexpr int kBBytes = BN * 128;      // BN x 64 K (K-major) or 64 K x BN (N-major)
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ GemmBars bars;
    __shared__ uint32_t tmem_base;
    __shared__ int fail;
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~static_cast<uintptr_t>(1023));
    unsigned char *sa = smem;                          // kStages x A tile
    unsigned char *sb = smem + kStages * kABytes;      // kStages x B tile
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int m0 = blockIdx.x * kTileM, n0 = blockIdx.y * BN, g = blockIdx.z;
    const int nk = (p.K + 63) / 64;
    const uint64_t lim = kWaitLimitNs;

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&bars.full_a[s], 4);
            mbar_init(&bars.full_b[s], 1);
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
    const uint32_t tmem = tmem_base;
    auto bail = [&]() {
        record_status(p.status, kStatusTimeout);
        fail = 1;
    };

    if (warp == 0) {
        // ---- weight tiles by TMA
        for (int c = 0; c < nk; ++c) {
            const int s = c % kStages, round = c / kStages;
            if (round >= 1 && !__all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.empty[s]), (round - 1) & 1, lim))) {
                if (lane == 0) bail();
                break;
            }
            if (lane == 0) {
                const uint32_t fb = smem_u32(&bars.full_b[s]);
                tc::mbar_arrive_expect_tx(fb, kBBytes);
                const uint32_t dst = smem_u32(sb + s * kBBytes);
                if (NMAJ) {
                    // rows = K of group g, columns = N: one 64 x 64 box per 64 columns
                    for (int j = 0; j < BN / 64; ++j)
                        tc::tma_load_2d(dst + j * 64 * 128, &map_b, n0 + 64 * j, g * p.K + 64 * c, fb);
                } else {
                    tc::tma_load_2d(dst, &map_b, 64 * c, g * p.N + n0, fb);
                }
            }
            __syncwarp();
        }
    } else if (warp == 1) {
        // ---- MMA issuer (converged warp, one elected lane issues)
        const uint32_t idesc = tc::idesc_bf16_f32(kTileM, BN, false, NMAJ);
        const uint64_t da = tc::smem_desc(0, 16, 1024, tc::kSwizzle128B);
        const uint64_t db = NMAJ ? tc::smem_desc(0, 64 * 128, 1024, tc::kSwizzle128B)
                                 : tc::smem_desc(0, 16, 1024, tc::kSwizzle128B);
        auto with_addr = [](uint64_t tmpl, uint32_t saddr) {
            return tmpl | static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
        };
        bool ok = true;
        for (int c = 0; c < nk && ok; ++c) {
            const int s = c % kStages, par = (c / kStages) & 1;
            ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.full_b[s]), par, lim) &&
                                             mbar_wait(smem_u32(&bars.full_a[s]), par, lim));
            if (!ok) break;
            tc::fence_after_sync();
            const uint32_t a_base = smem_u32(sa + s * kABytes), b_base = smem_u32(sb + s * kBBytes);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
                const uint32_t b_addr = NMAJ ? b_base + kk * 16 * 128 : b_base + kk * 32;
                tc::mma_bf16_elect(tmem, with_addr(da, a_base + kk * 32), with_addr(db, b_addr), idesc,
                                   (c | kk) != 0);
            }
            tc::commit_elect(smem_u32(&bars.empty[s]));
        }
        if (!ok && lane == 0) bail();
        tc::commit_elect(smem_u32(&bars.done));
    } else {
        // ---- A rows: thread r of warps 2..5 owns tile row r; 64 K values per stage
        const int r = tid - 64;
        const int m = m0 + r;
        const bool valid = m < p.M;
        const int64_t row = valid ? phys_row(p, g, m) : 0;
        for (int c = 0; c < nk; ++c) {
            const int s = c % kStages, round = c / kStages;
            if (round >= 1 && !__all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.empty[s]), (round - 1) & 1, lim))) {
                if (lane == 0) bail();
                break;
            }
            uint4 packed[8];
            const int k0 = 64 * c;
            if (valid && k0 + 64 <= p.K) {
                if (p.a_f32) {
                    const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(p.A) + row * p.lda + k0);
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const float4 x = src[2 * j], y = src[2 * j + 1];
                        const __nv_bfloat162 b0 = __floats2bfloat162_rn(x.x, x.y), b1 = __floats2bfloat162_rn(x.z, x.w);
                        const __nv_bfloat162 b2 = __floats2bfloat162_rn(y.x, y.y), b3 = __floats2bfloat162_rn(y.z, y.w);
                        packed[j] = make_uint4(*reinterpret_cast<const uint32_t *>(&b0), *reinterpret_cast<const uint32_t *>(&b1),
                                               *reinterpret_cast<const uint32_t *>(&b2), *reinterpret_cast<const uint32_t *>(&b3));
                    }
                } else {
                    const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(p.A) + row * p.lda + k0);
#pragma unroll
                    for (int j = 0; j < 8; ++j) packed[j] = src[j];
                }
            } else {
                // rows past M, or the ragged end of K: element-wise, zero beyond
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    uint32_t u[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int k = k0 + 8 * j + 2 * e;
                        const float x0 = (valid && k < p.K) ? a_value(p, row, k) : 0.f;
                        const float x1 = (valid && k + 1 < p.K) ? a_value(p, row, k + 1) : 0.f;
                        const __nv_bfloat162 b = __floats2bfloat162_rn(x0, x1);
                        u[e] = *reinterpret_cast<const uint32_t *>(&b);
                    }
                    packed[j] = make_uint4(u[0], u[1], u[2], u[3]);
                }
            }
            uint4 *dst = reinterpret_cast<uint4 *>(sa + s * kABytes + r * 128);
#pragma unroll
            for (int j = 0; j < 8; ++j) dst[j ^ (r & 7)] = packed[j];
            tc::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(smem_u32(&bars.full_a[s]));
        }
        // ---- epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31
        const bool ok = __all_sync(0xffffffffu, mbar_wait(smem_u32(&bars.done), 0, lim));
        if (!ok) {
            if (lane == 0) bail();
        } else if (!fail) {
            tc::fence_after_sync();
            const int q = warp & 3;
            const int me = m0 + q * 32 + lane;
            const uint32_t t_lane = tmem + (static_cast<uint32_t>(q * 32) << 16);
            const int64_t orow = me < p.M ? phys_row(p, g, me) : 0;
#pragma unroll 1
            for (int j = 0; j < BN; j += 16) {
                uint32_t v[16];
                tc::ld_32x32b_x16(t_lane + j, v);
                tc::wait_ld();
                const int n = n0 + j;
                if (me >= p.M || n >= p.N) continue;
                uint16_t *dst = static_cast<uint16_t *>(p.C) + orow * p.ldc + n;
                if (n + 16 <= p.N) {
                    uint32_t w[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const __nv_bfloat162 b = __floats2bfloat162_rn(__uint_as_float(v[2 * e]), __uint_as_float(v[2 * e + 1]));
                        w[e] = *reinterpret_cast<const uint32_t *>(&b);
                    }
                    reinterpret_cast<uint4 *>(dst)[0] = make_uint4(w[0], w[1], w[2], w[3]);
                    reinterpret_cast<uint4 *>(dst)[1] = make_uint4(w[4], w[5], w[6], w[7]);
                } else {
                    for (int e = 0; e < 16 && n + e < p.N; ++e)
                        dst[e] = __bfloat16_as_ushort(__float2bfloat16_rn(__uint_as_float(v[e])));
                }
            }
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, BN < 32 ? 32 : BN);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 g_encode_gemm = nullptr;

template <int BN, bool NMAJ>
cudaError_t launch_tc(const GroupGemm &p, cudaStream_t st)
{
    if (!g_encode_gemm) {
        cudaDriverEntryPointQueryResult q;
        void *fn = nullptr;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) return e != cudaSuccess ? e : cudaErrorNotSupported;
        g_encode_gemm = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    CUtensorMap mb;
    cuuint64_t dims[2], strides[1];
    cuuint32_t box[2], es[2] = {1, 1};
    if (NMAJ) {  // [G K rows][N columns]
        dims[0] = static_cast<cuuint64_t>(p.N);
        dims[1] = static_cast<cuuint64_t>(p.G) * p.K;
        strides[0] = static_cast<cuuint64_t>(p.N) * 2;
        box[0] = 64;
        box[1] = 64;
    } else {     // [G N rows][K columns]
        dims[0] = static_cast<cuuint64_t>(p.K);
        dims[1] = static_cast<cuuint64_t>(p.G) * p.N;
        strides[0] = static_cast<cuuint64_t>(p.K) * 2;
        box[0] = 64;
        box[1] = BN;
    }
    CUresult r = g_encode_gemm(&mb, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(p.B), dims, strides, box, es,
                               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    const size_t smem = 1024 + static_cast<size_t>(kStages) * (kTileM * 128 + BN * 128);
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, NMAJ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    dim3 grid((p.M + kTileM - 1) / kTileM, (p.N + BN - 1) / BN, p.G);
    gemm_tc_kernel<BN, NMAJ><<<grid, kGemmThreads, smem, st>>>(p, mb);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_group_gemm(const GroupGemm &p, cudaStream_t st)
{
    if (p.M <= 0 || p.N <= 0 || p.G <= 0) return cudaSuccess;
    const size_t smem = static_cast<size_t>(p.M) * p.K * 4;
    if (!p.b_nmajor && p.M <= 32 && p.K >= 1024 && smem <= 160 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(small_kmajor_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        small_kmajor_kernel<<<dim3((p.N + kSmallCols - 1) / kSmallCols, p.G), 32 * kSmallWarps, smem, st>>>(p);
        return cudaGetLastError();
    }
    // column tile: 64 for narrow outputs, else 128 (more CTAs than 256 would give)
    if (p.b_nmajor) return p.N <= 64 ? launch_tc<64, true>(p, st) : launch_tc<128, true>(p, st);
    return p.N <= 64 ? launch_tc<64, false>(p, st) : launch_tc<128, false>(p, st);
}

}  // namespace gbmla
