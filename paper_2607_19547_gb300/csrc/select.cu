// Step 3 of the composition path: top-rho selection (ChronoStitch Sec. 2).
//
// One CTA of 1024 threads (the candidate scores are a few hundred KB and stay
// in L2).  Scores map to order-preserving 32-bit keys; four MSB-first radix
// passes over 8-bit digits find K*, the k-th largest key, and how many keys
// equal to K* belong to the top k (the lowest-index ones: the tie-break).  A
// final pass in index order writes the selected indices with a block-wide
// prefix count, so the output is ascending without a sort.
#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;

// Order-preserving key of an fp32 bit pattern u (scores are read as raw 32-bit
// words, never as floats, so every NaN payload and sign survives).
__device__ __forceinline__ uint32_t order_key(uint32_t u) {
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__global__ void __launch_bounds__(kThreads, 1)
select_kernel(const uint32_t *__restrict__ score, int n, int k, int idx_base, int *__restrict__ out) {
    __shared__ uint32_t hist[kWarps][256];
    __shared__ uint32_t total[256];
    __shared__ uint32_t s_digit, s_krem;
    __shared__ uint32_t wcnt[kWarps][2];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    if (k >= n) {   // everything is selected, in index order
        for (int i = tid; i < n; i += kThreads) out[i] = idx_base + i;
        return;
    }
    uint32_t prefix = 0, pmask = 0, krem = static_cast<uint32_t>(k);
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        for (int i = tid; i < kWarps * 256; i += kThreads) (&hist[0][0])[i] = 0;
        __syncthreads();
        for (int i = tid; i < n; i += kThreads) {
            const uint32_t key = order_key(__ldg(score + i));
            if ((key & pmask) == prefix) atomicAdd(&hist[warp][(key >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (tid < 256) {
            uint32_t c = 0;
#pragma unroll 8
            for (int w = 0; w < kWarps; ++w) c += hist[w][tid];
            total[tid] = c;
        }
        __syncthreads();
        if (warp == 0) {
            // lane l scans bins 255-8l down to 248-8l; lanes in order cover bins high -> low
            uint32_t cnt[8], local = 0;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                cnt[j] = total[255 - 8 * lane - j];
                local += cnt[j];
            }
            uint32_t incl = local;
#pragma unroll
            for (int o = 1; o < 32; o *= 2) {
                const uint32_t up = __shfl_up_sync(0xFFFFFFFFu, incl, o);
                if (lane >= o) incl += up;
            }
            uint32_t above = incl - local;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                if (above < krem && above + cnt[j] >= krem) {
                    s_digit = 255u - 8u * lane - j;
                    s_krem = krem - above;
                }
                above += cnt[j];
            }
        }
        __syncthreads();
        prefix |= s_digit << shift;
        pmask |= 0xFFu << shift;
        krem = s_krem;
        __syncthreads();
    }
    // prefix = K*; krem = how many keys equal to K* are selected (lowest indices first)
    const uint32_t kstar = prefix;
    uint32_t run_gt = 0, run_eq = 0;
    const uint32_t lt_mask = (1u << lane) - 1u;
    for (int base = 0; base < n; base += kThreads) {
        const int i = base + tid;
        const uint32_t key = (i < n) ? order_key(__ldg(score + i)) : 0u;
        const bool gt = (i < n) && key > kstar;
        const bool eq = (i < n) && key == kstar;
        const uint32_t bg = __ballot_sync(0xFFFFFFFFu, gt);
        const uint32_t be = __ballot_sync(0xFFFFFFFFu, eq);
        if (lane == 0) {
            wcnt[warp][0] = __popc(bg);
            wcnt[warp][1] = __popc(be);
        }
        __syncthreads();
        uint32_t pre_g = 0, pre_e = 0, tot_g = 0, tot_e = 0;
        for (int w = 0; w < kWarps; ++w) {   // broadcast reads; 32 entries
            const uint32_t cg = wcnt[w][0], ce = wcnt[w][1];
            if (w < warp) { pre_g += cg; pre_e += ce; }
            tot_g += cg;
            tot_e += ce;
        }
        const uint32_t eq_before = run_eq + pre_e + __popc(be & lt_mask);
        const uint32_t gt_before = run_gt + pre_g + __popc(bg & lt_mask);
        if (gt || (eq && eq_before < krem)) {
            const uint32_t pos = gt_before + min(eq_before, krem);
            out[pos] = idx_base + i;
        }
        run_gt += tot_g;
        run_eq += tot_e;
        __syncthreads();
    }
}

}  // namespace

cudaError_t launch_select(const float *score, int n, int k, int idx_base, int *out,
                          cudaStream_t s) {
    if (k == 0 || n == 0) return cudaSuccess;
    select_kernel<<<1, kThreads, 0, s>>>(reinterpret_cast<const uint32_t *>(score), n, k, idx_base,
                                         out);
    return cudaGetLastError();
}

}  // namespace cs
