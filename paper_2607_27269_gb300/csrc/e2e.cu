// mla_e2e_loss: forward value of the E2E functional-reconstruction loss of one
// layer (Sec. 4.1), the masked mean-squared error between the converted MLA
// block's post-W_O output and the frozen original block's:
//   L = sum_t M_t sum_d (A_MLA[t, d] - A_orig[t, d])^2 / (D sum_t M_t).
// One cluster of kCl CTAs: CTA c sums the rows [c R / kCl, (c + 1) R / kCl),
// each thread a fixed set of 8-element vectors (fp32 within a vector, fp64
// across); the CTAs push their (sum, counted rows) into rank 0, which adds them
// in rank order, so the result is the same bits on every run.
#include "common.cuh"
#include "internal.h"
#include "tc.cuh"

namespace gbmla {
namespace {

constexpr int kCl = 8;
constexpr int kE2eThreads = 512;

__global__ void __launch_bounds__(kE2eThreads) e2e_loss_kernel(int rows, int hidden, const uint16_t *__restrict__ a,
                                                              const uint16_t *__restrict__ b,
                                                              const uint8_t *__restrict__ mask, float *loss)
{
    __shared__ double red[kE2eThreads / 32];
    __shared__ double s_num[kCl], s_den[kCl];  // rank 0's copies are read
    // every CTA of the cluster must have started before one writes another's shared memory
    asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    griddep_wait();
    griddep_launch_dependents();
    const int rank = blockIdx.x;
    const int r0 = static_cast<int>(static_cast<int64_t>(rank) * rows / kCl);
    const int r1 = static_cast<int>(static_cast<int64_t>(rank + 1) * rows / kCl);
    const int vpr = hidden / 8;  // 8-element vectors per row
    double acc = 0.0;
    const int64_t nvec = static_cast<int64_t>(r1 - r0) * vpr;
    for (int64_t v = threadIdx.x; v < nvec; v += kE2eThreads) {
        const int t = r0 + static_cast<int>(v / vpr);
        if (mask && !mask[t]) continue;
        const int64_t off = static_cast<int64_t>(t) * hidden + (v % vpr) * 8;
        const uint4 x = *reinterpret_cast<const uint4 *>(a + off), y = *reinterpret_cast<const uint4 *>(b + off);
        const uint32_t xa[4] = {x.x, x.y, x.z, x.w}, ya[4] = {y.x, y.y, y.z, y.w};
        float s = 0.f;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float d0 = __uint_as_float(xa[e] << 16) - __uint_as_float(ya[e] << 16);
            const float d1 = __uint_as_float(xa[e] & 0xffff0000u) - __uint_as_float(ya[e] & 0xffff0000u);
            s = fmaf(d0, d0, s);
            s = fmaf(d1, d1, s);
        }
        acc += s;
    }
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
    if (threadIdx.x == 0) {
        double num = 0.0, den = 0.0;
        for (int w = 0; w < kE2eThreads / 32; ++w) num += red[w];
        for (int t = r0; t < r1; ++t) den += (!mask || mask[t]) ? 1.0 : 0.0;
        uint32_t remote;
        asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(&s_num[rank])), "r"(0));
        asm volatile("st.shared::cluster.f64 [%0], %1;" ::"r"(remote), "d"(num) : "memory");
        asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(&s_den[rank])), "r"(0));
        asm volatile("st.shared::cluster.f64 [%0], %1;" ::"r"(remote), "d"(den) : "memory");
    }
    tc::cluster_sync();
    if (rank == 0 && threadIdx.x == 0) {
        double num = 0.0, den = 0.0;
        for (int c = 0; c < kCl; ++c) {
            num += s_num[c];
            den += s_den[c];
        }
        *loss = den > 0.0 ? static_cast<float>(num / (static_cast<double>(hidden) * den)) : 0.f;
    }
}

}  // namespace

cudaError_t launch_e2e_loss(int rows, int hidden, const void *a_mla, const void *a_orig, const uint8_t *mask,
                            float *loss, cudaStream_t st)
{
    return launch_dependent(e2e_loss_kernel, dim3(kCl), dim3(kE2eThreads), 0, st, kCl, rows, hidden,
                            static_cast<const uint16_t *>(a_mla), static_cast<const uint16_t *>(a_orig), mask, loss);
}

}  // namespace gbmla
