// Step 2 of the composition path: key-deviation score (ChronoStitch, Eq. 5).
//
// One warp per candidate token.  Lane b owns 8-element blocks b, b+32, ...;
// it loads each block with 16-byte vector loads, forms the block sum
// ((q0+q1)+(q2+q3))+((q4+q5)+(q6+q7)) of q_j = (a_j - b_j)^2, folds its own
// blocks with the strides >= 32 of the fixed halving order, and the warp
// finishes strides 16..1 with an xor butterfly (s[b] + s[b^m] = s[b] + s[b+m]
// for b < m, fp32 addition being commutative).  Blocks beyond the row length
// are +0.  The order is the one the header documents, so the result is
// bit-reproducible.  HBM-bound: two key rows in, one fp32 out per token.
#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kWarpsPerCta = 8;

__device__ __forceinline__ float block8(const float (&a)[8], const float (&b)[8]) {
    float q[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float d = __fsub_rn(a[e], b[e]);
        q[e] = __fmul_rn(d, d);
    }
    return __fadd_rn(__fadd_rn(__fadd_rn(q[0], q[1]), __fadd_rn(q[2], q[3])),
                     __fadd_rn(__fadd_rn(q[4], q[5]), __fadd_rn(q[6], q[7])));
}

__device__ __forceinline__ void load8(const __nv_bfloat16 *p, float (&x)[8]) {
    const uint4 v = __ldg(reinterpret_cast<const uint4 *>(p));
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        x[2 * i] = bf16_lo(w[i]);
        x[2 * i + 1] = bf16_hi(w[i]);
    }
}

__device__ __forceinline__ void load8(const float *p, float (&x)[8]) {
    const float4 u = __ldg(reinterpret_cast<const float4 *>(p));
    const float4 v = __ldg(reinterpret_cast<const float4 *>(p + 4));
    x[0] = u.x; x[1] = u.y; x[2] = u.z; x[3] = u.w;
    x[4] = v.x; x[5] = v.y; x[6] = v.z; x[7] = v.w;
}

// NJ = blocks per lane after padding to a power of two (1 when fewer than 32 blocks).
template <typename T, int NJ>
__global__ void __launch_bounds__(kWarpsPerCta * 32)
score_kernel(const T *__restrict__ fresh, const T *__restrict__ cached, int n, int nblocks,
             long long fs, long long cst, float *__restrict__ out) {
    pdl_wait();   // inputs may come from the previous kernel of the stream
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const int row = blockIdx.x * kWarpsPerCta + (threadIdx.x >> 5);
    if (row >= n) return;
    const T *a = fresh + static_cast<long long>(row) * fs;
    const T *b = cached + static_cast<long long>(row) * cst;
    float s[NJ];
#pragma unroll
    for (int j = 0; j < NJ; ++j) {
        const int blk = lane + 32 * j;
        s[j] = 0.0f;
        if (blk < nblocks) {
            float x[8], y[8];
            load8(a + 8 * blk, x);
            load8(b + 8 * blk, y);
            s[j] = block8(x, y);
        }
    }
#pragma unroll
    for (int m = NJ / 2; m >= 1; m /= 2) {
#pragma unroll
        for (int j = 0; j < m; ++j) s[j] = __fadd_rn(s[j], s[j + m]);
    }
    float v = s[0];
#pragma unroll
    for (int m = 16; m >= 1; m /= 2) v = __fadd_rn(v, __shfl_xor_sync(0xFFFFFFFFu, v, m));
    if (lane == 0) out[row] = v;
}

template <typename T>
cudaError_t launch_typed(const void *fresh, const void *cached, int n, int E, long long fs,
                         long long cst, float *out, cudaStream_t s) {
    const int nblocks = E / 8;
    int P = 1;
    while (P < nblocks) P *= 2;
    const int NJ = P <= 32 ? 1 : P / 32;
    const dim3 grid((n + kWarpsPerCta - 1) / kWarpsPerCta);
    const T *f = static_cast<const T *>(fresh);
    const T *c = static_cast<const T *>(cached);
    switch (NJ) {
        case 1: return launch_pdl(score_kernel<T, 1>, grid, dim3(kWarpsPerCta * 32), 0, s, f, c, n, nblocks, fs, cst, out);
        case 2: return launch_pdl(score_kernel<T, 2>, grid, dim3(kWarpsPerCta * 32), 0, s, f, c, n, nblocks, fs, cst, out);
        case 4: return launch_pdl(score_kernel<T, 4>, grid, dim3(kWarpsPerCta * 32), 0, s, f, c, n, nblocks, fs, cst, out);
        case 8: return launch_pdl(score_kernel<T, 8>, grid, dim3(kWarpsPerCta * 32), 0, s, f, c, n, nblocks, fs, cst, out);
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_score(const void *fresh, const void *cached, cs_dtype dt, int n, int E,
                         long long fresh_stride, long long cached_stride, float *out,
                         cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    if (dt == CS_DTYPE_BF16)
        return launch_typed<__nv_bfloat16>(fresh, cached, n, E, fresh_stride, cached_stride, out, s);
    return launch_typed<float>(fresh, cached, n, E, fresh_stride, cached_stride, out, s);
}

}  // namespace cs
