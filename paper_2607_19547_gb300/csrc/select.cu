// Step 3 of the composition path: top-rho selection (ChronoStitch Sec. 2).
//
// One CTA of 1024 threads (the candidate scores are a few hundred KB at most and
// stay in L2).  Scores map to order-preserving 32-bit keys.  Thread t owns the
// contiguous candidate range [t*per, (t+1)*per); up to 16 keys per thread stay
// in registers, larger inputs are re-read from L2 in every pass (the histogram
// passes read them interleaved and coalesced, eight loads in flight).  Up to three
// MSB-first radix passes over 11-, 11- and 10-bit digits (one shared 2048-bin
// histogram, shared-memory atomic increments) find K*, the k-th largest key, and how
// many keys equal to K* belong to the top k (the lowest-index ones: the
// tie-break); they stop early once every key left in K*'s bin is taken, and the
// resolved prefix of K* then stands for it.  One block-wide scan of the per-thread (greater, equal) counts
// then gives every selected index its output position, so the output is
// ascending without a sort.
#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
constexpr int kBins = 2048;
constexpr int kRegKeys = 16;   // keys per thread held in registers (n <= 16384)

// Order-preserving key of an fp32 bit pattern u (scores are read as raw 32-bit
// words, never as floats, so every NaN payload and sign survives).
__device__ __forceinline__ uint32_t order_key(uint32_t u) {
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// hist[d] += 1 for every lane with `active`.  Plain shared-memory atomics: lanes
// that share a digit (scores of one binade often do) were measured faster this way
// than aggregated with __match_any_sync first (10.7 / 18.3 / 59.7 us against 12.6 /
// 29.0 / 112 us for 3 072 / 15 360 / 64 512 candidates).
__device__ __forceinline__ void hist_add(uint32_t *hist, uint32_t d, bool active) {
    if (active) atomicAdd(&hist[d], 1u);
}

// Block-wide inclusive scan of v (all 1024 threads call; wsum holds 32 words).
// Callers separate two uses of wsum with a barrier.
template <typename T>
__device__ __forceinline__ T block_incl_scan(T v, T *wsum) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 1; o < 32; o *= 2) {
        const T y = __shfl_up_sync(0xFFFFFFFFu, v, o);
        if (lane >= o) v += y;
    }
    if (lane == 31) wsum[warp] = v;
    __syncthreads();
    if (warp == 0) {
        T w = wsum[lane];
#pragma unroll
        for (int o = 1; o < 32; o *= 2) {
            const T y = __shfl_up_sync(0xFFFFFFFFu, w, o);
            if (lane >= o) w += y;
        }
        wsum[lane] = w;
    }
    __syncthreads();
    return warp > 0 ? v + wsum[warp - 1] : v;
}

// KPT > 0: exactly KPT keys per thread in registers; KPT == 0: per keys per
// thread read from global memory in every pass.
template <int KPT>
__global__ void __launch_bounds__(kThreads, 1)
select_kernel(const uint32_t *__restrict__ score, int n, int k, int idx_base, int per,
              int *__restrict__ out) {
    pdl_wait();   // inputs may come from the previous kernel of the stream
    pdl_trigger();
    __shared__ uint32_t hist[kBins];
    __shared__ unsigned long long wsum[kWarps];
    __shared__ uint32_t s_digit, s_krem, s_done;
    const int tid = threadIdx.x;

    if (k >= n) {   // everything is selected, in index order
        for (int i = tid; i < n; i += kThreads) out[i] = idx_base + i;
        return;
    }
    const int i0 = tid * per;
    const int cnt = max(0, min(per, n - i0));
    uint32_t reg[KPT > 0 ? KPT : 1];
    if (KPT > 0) {
#pragma unroll
        for (int i = 0; i < (KPT > 0 ? KPT : 1); ++i)
            reg[i] = i < cnt ? order_key(__ldg(score + i0 + i)) : 0u;
    }
    auto key_at = [&](int i) -> uint32_t {
        if (KPT > 0) return reg[i];
        return order_key(__ldg(score + i0 + i));
    };

    uint32_t prefix = 0, pmask = 0, krem = static_cast<uint32_t>(k);
#pragma unroll 1
    for (int pass = 0; pass < 3; ++pass) {
        const int shift = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
        const uint32_t dmask = pass == 2 ? 0x3FFu : 0x7FFu;
        for (int b = tid; b < kBins; b += kThreads) hist[b] = 0;
        __syncthreads();
        if (KPT > 0) {
#pragma unroll
            for (int i = 0; i < (KPT > 0 ? KPT : 1); ++i) {
                const uint32_t key = reg[i];
                hist_add(hist, (key >> shift) & dmask, i < cnt && (key & pmask) == prefix);
            }
        } else {
            // the histogram does not care which thread counts which key: read the keys
            // interleaved (coalesced), eight loads in flight before their increments
            const int rounds = (n + kThreads * 8 - 1) / (kThreads * 8);   // uniform
            for (int rr = 0; rr < rounds; ++rr) {
                uint32_t kb[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int i = (rr * 8 + u) * kThreads + tid;
                    kb[u] = i < n ? order_key(__ldg(score + i)) : 0u;
                }
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int i = (rr * 8 + u) * kThreads + tid;
                    hist_add(hist, (kb[u] >> shift) & dmask, i < n && (kb[u] & pmask) == prefix);
                }
            }
        }
        __syncthreads();
        // thread t holds bins 2047-2t and 2046-2t; an inclusive scan from the top
        // finds the bin in which the k-th largest key falls
        const uint32_t hi = hist[kBins - 1 - 2 * tid], lo = hist[kBins - 2 - 2 * tid];
        const unsigned long long incl =
            block_incl_scan<unsigned long long>(static_cast<unsigned long long>(hi + lo), wsum);
        const unsigned long long above = incl - (hi + lo);
        if (above < krem && incl >= krem) {
            // the bin holding the k-th largest key; when every key left in it is taken,
            // the remaining digits cannot change the selection and the passes stop
            if (above + hi >= krem) {
                s_digit = static_cast<uint32_t>(kBins - 1 - 2 * tid);
                s_krem = krem - static_cast<uint32_t>(above);
                s_done = hi == s_krem;
            } else {
                s_digit = static_cast<uint32_t>(kBins - 2 - 2 * tid);
                s_krem = krem - static_cast<uint32_t>(above) - hi;
                s_done = lo == s_krem;
            }
        }
        __syncthreads();
        prefix |= s_digit << shift;
        pmask |= dmask << shift;
        krem = s_krem;
        if (s_done) break;   // uniform; nothing shared is written again before it is read
        __syncthreads();     // s_digit / wsum are rewritten by the next pass
    }
    // prefix = the resolved high bits of K* (all of K* after three passes) and pmask
    // their mask; krem = how many keys with that prefix are selected (lowest indices first;
    // all of them when the passes stopped early)
    const uint32_t kstar = prefix;
    uint32_t gt = 0, eq = 0;
    if (KPT > 0) {
#pragma unroll
        for (int i = 0; i < (KPT > 0 ? KPT : 1); ++i) {
            gt += (i < cnt && (reg[i] & pmask) > kstar);
            eq += (i < cnt && (reg[i] & pmask) == kstar);
        }
    } else {
        for (int c0 = 0; c0 < cnt; c0 += 8) {   // eight loads in flight
            uint32_t kb[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) kb[u] = c0 + u < cnt ? (key_at(c0 + u) & pmask) : 0u;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                gt += c0 + u < cnt && kb[u] > kstar;
                eq += c0 + u < cnt && kb[u] == kstar;
            }
        }
    }
    const unsigned long long mine = (static_cast<unsigned long long>(gt) << 32) | eq;
    const unsigned long long before = block_incl_scan<unsigned long long>(mine, wsum) - mine;
    const uint32_t gt_before = static_cast<uint32_t>(before >> 32);
    uint32_t eq_seen = static_cast<uint32_t>(before & 0xFFFFFFFFu);
    uint32_t pos = gt_before + min(eq_seen, krem);
    if (KPT > 0) {
#pragma unroll
        for (int i = 0; i < (KPT > 0 ? KPT : 1); ++i) {
            const uint32_t key = reg[i] & pmask;
            if (i < cnt && (key > kstar || (key == kstar && eq_seen++ < krem)))
                out[pos++] = idx_base + i0 + i;
        }
    } else {
        for (int c0 = 0; c0 < cnt; c0 += 8) {
            uint32_t kb[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) kb[u] = c0 + u < cnt ? (key_at(c0 + u) & pmask) : 0u;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const uint32_t key = kb[u];
                if (c0 + u < cnt && (key > kstar || (key == kstar && eq_seen++ < krem)))
                    out[pos++] = idx_base + i0 + c0 + u;
            }
        }
    }
}

}  // namespace

cudaError_t launch_select(const float *score, int n, int k, int idx_base, int *out,
                          cudaStream_t s) {
    if (k == 0 || n == 0) return cudaSuccess;
    const uint32_t *keys = reinterpret_cast<const uint32_t *>(score);
    const int per = (n + kThreads - 1) / kThreads;
    if (per <= 4) {
        return launch_pdl(select_kernel<4>, dim3(1), dim3(kThreads), 0, s, keys, n, k, idx_base, 4, out);
    } else if (per <= kRegKeys) {
        return launch_pdl(select_kernel<kRegKeys>, dim3(1), dim3(kThreads), 0, s, keys, n, k, idx_base,
                          kRegKeys, out);
    } else {
        return launch_pdl(select_kernel<0>, dim3(1), dim3(kThreads), 0, s, keys, n, k, idx_base, per, out);
    }
    return cudaGetLastError();
}

}  // namespace cs
