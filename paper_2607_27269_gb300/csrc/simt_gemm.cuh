// A plain CUDA-core tile GEMM used by the small projections until they move
// to the tensor cores: C[m, n] = sum_k A(m, k) * B(n, k), fp32 accumulation.
#pragma once

#include "common.cuh"

namespace gbmla {

// One 64x64 output tile per 256-thread block, K in steps of 16.  The three
// functors map logical indices to loads and the store; loads outside
// [0,M)x[0,K) or [0,N)x[0,K) read as zero.
template <class LoadA, class LoadB, class Store>
__device__ __forceinline__ void simt_gemm_64x64(int m0, int n0, int M, int N, int K, LoadA load_a,
                                                LoadB load_b, Store store)
{
    __shared__ float As[16][68];
    __shared__ float Bs[16][68];
    const int tid = threadIdx.x;
    const int tm = (tid >> 4) * 4, tn = (tid & 15) * 4;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < K; k0 += 16) {
        for (int e = tid; e < 64 * 16; e += 256) {
            const int mm = e >> 4, kk = e & 15;
            const int gk = k0 + kk;
            const int gm = m0 + mm, gn = n0 + mm;
            As[kk][mm] = (gm < M && gk < K) ? load_a(gm, gk) : 0.f;
            Bs[kk][mm] = (gn < N && gk < K) ? load_b(gn, gk) : 0.f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            float av[4], bv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) av[i] = As[kk][tm + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tn + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j)
            if (m0 + tm + i < M && n0 + tn + j < N) store(m0 + tm + i, n0 + tn + j, acc[i][j]);
}

}  // namespace gbmla
