// Step 3 of the composition path: top-rho selection (ChronoStitch Sec. 2).
//
// Scores map to order-preserving 32-bit keys; the k largest keys win, equal keys
// rank the lower index first, and the output is the selected indices in
// ascending order.  Up to 8192 scores: one CTA (select_small_kernel below).  Beyond
// that: exact radix select over one thread-block cluster of C CTAs (C = 2, 4, 8 or 16,
// sized from n; 1 where the device cannot co-schedule a cluster):
//   - CTA r owns the contiguous candidate range [r*span, (r+1)*span) and thread t
//     of it the contiguous range [t*per, (t+1)*per) inside that; up to 16 keys per
//     thread stay in registers (16-byte loads), larger inputs are re-read in every
//     pass;
//   - up to three MSB-first passes over 11-, 11- and 10-bit digits find K*, the
//     k-th largest key, and how many keys equal to K* are taken (the lowest-index
//     ones).  A pass: every CTA counts its own keys that match the digits resolved
//     so far into a 2048-bin histogram in its shared memory and sums it over 64
//     groups of 32 bins; after one cluster barrier every CTA reads the C x 64 group
//     sums through distributed shared memory (spread over its threads), finds the
//     group that holds the k-th key with a warp-wide scan, then reads that group's
//     32 bins from the C CTAs and finds the bin the same way.  Every CTA takes the
//     same decision from the same counts.  The histograms are double-buffered by pass parity, so a CTA never
//     clears a buffer that another CTA may still read.  The passes stop once every
//     key left in K*'s bin is taken;
//   - one block-wide scan of the per-thread (greater, equal) counts, plus the
//     counts of the CTAs before it (read from their shared memory), gives every
//     thread its first output position, so the output is ascending without a sort.
// The cluster barriers are hardware barriers that every thread of every CTA
// reaches the same number of times (the decisions are identical in every CTA); a
// final barrier keeps each CTA's shared memory alive until the others have read it.
// No global memory besides the scores and the output is used.
#include <algorithm>
#include <mutex>

#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kNT = 512;          // threads per CTA
constexpr int kWarps = kNT / 32;
constexpr int kBins = 2048;
constexpr int kFine = 32;                  // bins per group
constexpr int kGroups = kBins / kFine;     // 64 groups
constexpr int kMaxCluster = 16;

// Order-preserving key of an fp32 bit pattern u (scores are read as raw 32-bit
// words, never as floats, so every NaN payload and sign survives).
__device__ __forceinline__ uint32_t order_key(uint32_t u) {
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Cluster-wide barrier: release (this CTA's shared-memory writes) / acquire.
__device__ __forceinline__ void cluster_arrive() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
    asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_sync() {
    cluster_arrive();
    cluster_wait();
}

// Address of `p` (this CTA's shared memory) in the shared memory of CTA `rank`.
__device__ __forceinline__ uint32_t dsmem_addr(const void *p, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
    return r;
}
__device__ __forceinline__ uint32_t dsmem_ld(uint32_t addr) {
    uint32_t v;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}
__device__ __forceinline__ unsigned long long dsmem_ld64(uint32_t addr) {
    unsigned long long v;
    asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(addr) : "memory");
    return v;
}

// Block-wide inclusive scan of v (all kNT threads call; wsum holds kWarps words).
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
        T w = lane < kWarps ? wsum[lane] : T(0);
#pragma unroll
        for (int o = 1; o < kWarps; o *= 2) {
            const T y = __shfl_up_sync(0xFFFFFFFFu, w, o);
            if (lane >= o) w += y;
        }
        if (lane < kWarps) wsum[lane] = w;
    }
    __syncthreads();
    return warp > 0 ? v + wsum[warp - 1] : v;
}

struct SelShared {
    uint32_t hist[2][kBins];            // per-pass histograms (double-buffered by pass parity)
    uint32_t coarse[2][kGroups];        // their sums over groups of kFine consecutive bins
    unsigned long long wsum[kWarps];    // block scan scratch
    unsigned long long cta_counts;      // this CTA's (greater << 32 | equal) in the final phase
    unsigned long long s_before;        // counts of the CTAs before this one
    uint32_t part[kNT];                 // per-thread partial sums of a decision step
    uint32_t s_group, s_above, s_hit, s_cnt;   // the pass's decision
};

// Inclusive scan over the 32 lanes of a warp.
__device__ __forceinline__ uint32_t warp_incl_scan(uint32_t v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 1; o < 32; o *= 2) {
        const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, v, o);
        if (lane >= o) v += y;
    }
    return v;
}

// KPT > 0: exactly KPT keys per thread in registers (per == KPT); KPT == 0: `per`
// keys per thread (a multiple of 4) re-read from global memory in every pass.
// vec: the scores start 16-byte aligned (16-byte loads where a group of 4 is whole).
template <int KPT>
__global__ void __launch_bounds__(kNT, 1)
select_kernel(const uint32_t *__restrict__ score, int n, int k, int idx_base, int per, int vec,
              int *__restrict__ out) {
    pdl_wait();   // inputs may come from the previous kernel of the stream
    pdl_trigger();
    __shared__ __align__(16) SelShared sh;
    SelShared *s = &sh;
    const int t = threadIdx.x;
    const uint32_t C = gridDim.x;                // one cluster spans the grid
    const uint32_t r = C > 1 ? cluster_rank() : 0u;
    const long long i0 = (static_cast<long long>(r) * kNT + t) * per;   // first key of this thread
    const int cnt = static_cast<int>(max(0ll, min(static_cast<long long>(per), n - i0)));

    if (k >= n) {   // everything is selected, in index order (no barrier on this path)
        for (int i = 0; i < cnt; ++i) out[i0 + i] = idx_base + static_cast<int>(i0) + i;
        return;
    }

    // keys of this thread, four at a time
    auto load4 = [&](int c, uint32_t (&kb)[4]) {
        const long long g = i0 + 4 * c;
        if (vec && 4 * c + 3 < cnt) {
            const uint4 u = __ldg(reinterpret_cast<const uint4 *>(score + g));
            kb[0] = order_key(u.x); kb[1] = order_key(u.y);
            kb[2] = order_key(u.z); kb[3] = order_key(u.w);
        } else {
#pragma unroll
            for (int e = 0; e < 4; ++e) kb[e] = 4 * c + e < cnt ? order_key(__ldg(score + g + e)) : 0u;
        }
    };
    constexpr int kRegs = KPT > 0 ? KPT : 4;
    uint32_t reg[kRegs];
    if (KPT > 0) {
#pragma unroll
        for (int c = 0; c < kRegs / 4; ++c) {
            uint32_t kb[4];
            load4(c, kb);
#pragma unroll
            for (int e = 0; e < 4; ++e) reg[4 * c + e] = kb[e];
        }
    }
    // calls f(local index, key) for every key of this thread, in index order
    auto for_keys = [&](auto f) {
        if (KPT > 0) {
#pragma unroll
            for (int i = 0; i < kRegs; ++i)
                if (i < cnt) f(i, reg[i]);
        } else {
            for (int c = 0; 4 * c < cnt; ++c) {
                uint32_t kb[4];
                load4(c, kb);
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (4 * c + e < cnt) f(4 * c + e, kb[e]);
            }
        }
    };

    for (int j = t; j < 2 * kBins; j += kNT) (&s->hist[0][0])[j] = 0u;
    if (t < 2 * kGroups) (&s->coarse[0][0])[t] = 0u;
    if (t == 0) {   // defined even if a search found nothing (the counts rule that out)
        s->s_group = 0;
        s->s_above = 0;
        s->s_hit = 0;
        s->s_cnt = 0;
    }
    __syncthreads();

    // a word of this CTA's shared memory as seen in CTA c of the cluster (c == r: itself)
    auto rd = [&](const uint32_t *p, uint32_t c) -> uint32_t {
        return C == 1 ? *p : dsmem_ld(dsmem_addr(p, c));
    };
    const int lane = t & 31, warp = t >> 5;
    uint32_t prefix = 0, pmask = 0, krem = static_cast<uint32_t>(k);
#pragma unroll 1
    for (int pass = 0; pass < 3; ++pass) {
        const int shift = pass == 0 ? 21 : (pass == 1 ? 10 : 0);
        const uint32_t dmask = pass == 2 ? 0x3FFu : 0x7FFu;
        uint32_t *hist = s->hist[pass & 1];
        uint32_t *coarse = s->coarse[pass & 1];
        for_keys([&](int, uint32_t key) {
            if ((key & pmask) == prefix) atomicAdd(&hist[(key >> shift) & dmask], 1u);
        });
        __syncthreads();
        {   // group sums: thread t sums bins 4t..4t+3, eight threads make a group of 32
            const uint4 h4 = reinterpret_cast<const uint4 *>(hist)[t];
            uint32_t v = h4.x + h4.y + h4.z + h4.w;
            v += __shfl_xor_sync(0xFFFFFFFFu, v, 4);
            v += __shfl_xor_sync(0xFFFFFFFFu, v, 2);
            v += __shfl_xor_sync(0xFFFFFFFFu, v, 1);
            if ((t & 7) == 0) coarse[t >> 3] = v;
        }
        if (C > 1) {
            cluster_sync();
        } else {
            __syncthreads();
        }
        // every CTA has finished reading the other buffers (last pass): clear them
        for (int j = t; j < kBins; j += kNT) s->hist[(pass + 1) & 1][j] = 0u;
        if (t < kGroups) s->coarse[(pass + 1) & 1][t] = 0u;
        {   // cluster-wide group sums: thread t adds group t % 64 of CTAs t / 64, t / 64 + 8, ...
            uint32_t v = 0;
            for (uint32_t c = static_cast<uint32_t>(t / kGroups); c < C; c += kNT / kGroups)
                v += rd(&coarse[t % kGroups], c);
            s->part[t] = v;
        }
        __syncthreads();
        if (warp == 0) {
            // lane l holds groups 63 - 2l and 62 - 2l: lane order is descending digit order
            uint32_t ga = 0, gb = 0;
#pragma unroll
            for (int m = 0; m < kNT / kGroups; ++m) {
                ga += s->part[(kGroups - 1 - 2 * lane) + kGroups * m];
                gb += s->part[(kGroups - 2 - 2 * lane) + kGroups * m];
            }
            const uint32_t incl = warp_incl_scan(ga + gb);
            const uint32_t above = incl - ga - gb;
            if (above < krem && incl >= krem) {
                const bool hi = above + ga >= krem;
                s->s_group = static_cast<uint32_t>(hi ? kGroups - 1 - 2 * lane : kGroups - 2 - 2 * lane);
                s->s_above = hi ? above : above + ga;
            }
        }
        __syncthreads();
        const uint32_t grp = min(s->s_group, static_cast<uint32_t>(kGroups - 1));
        const uint32_t above_g = s->s_above;
        {   // the group's 32 bins in every CTA: thread t reads bin t % 32 of CTA t / 32
            const uint32_t c = static_cast<uint32_t>(t / kFine);
            s->part[t] = c < C ? rd(&hist[grp * kFine + lane], c) : 0u;
        }
        __syncthreads();
        if (warp == 0) {
            // lane l holds bin 31 - l of the group (descending digit order)
            uint32_t f = 0;
#pragma unroll
            for (int c = 0; c < kNT / kFine; ++c) f += s->part[(kFine - 1 - lane) + kFine * c];
            const uint32_t incl = warp_incl_scan(f);
            const uint32_t above = incl - f, want = krem - above_g;
            if (above < want && incl >= want) {
                s->s_hit = grp * kFine + static_cast<uint32_t>(kFine - 1 - lane);
                s->s_above = above_g + above;
                s->s_cnt = f;
            }
        }
        __syncthreads();
        // the digit of the k-th largest key among those with the resolved prefix; when
        // every key left in its bin is taken the remaining digits cannot change the
        // selection
        const uint32_t digit = s->s_hit;
        const uint32_t krem_new = krem - s->s_above;
        const bool done = s->s_cnt == krem_new;
        prefix |= digit << shift;
        pmask |= dmask << shift;
        krem = krem_new;
        __syncthreads();   // the decision words are rewritten in the next pass
        if (done) break;   // uniform across the cluster: every CTA took the same decision
    }

    // prefix = the resolved high bits of K* (all of K* after three passes), pmask their
    // mask; krem = how many keys with that prefix are selected (lowest indices first)
    const uint32_t kstar = prefix;
    uint32_t gt = 0, eq = 0;
    for_keys([&](int, uint32_t key) {
        gt += (key & pmask) > kstar;
        eq += (key & pmask) == kstar;
    });
    const unsigned long long mine = (static_cast<unsigned long long>(gt) << 32) | eq;
    const unsigned long long incl = block_incl_scan<unsigned long long>(mine, s->wsum);
    const unsigned long long before_t = incl - mine;
    if (t == kNT - 1) s->cta_counts = incl;
    unsigned long long before_cta = 0;
    if (C > 1) {
        cluster_sync();
        if (t < 32) {
            unsigned long long v = static_cast<uint32_t>(t) < r
                                       ? dsmem_ld64(dsmem_addr(&s->cta_counts, static_cast<uint32_t>(t)))
                                       : 0ull;
#pragma unroll
            for (int o = 16; o >= 1; o /= 2) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
            if (t == 0) s->s_before = v;
        }
        __syncthreads();
        before_cta = s->s_before;
        // this CTA reads no other CTA's shared memory after this point; the wait at the
        // end keeps its own alive until every CTA has read it
        asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
    }
    const unsigned long long before = before_cta + before_t;
    const uint32_t gt_before = static_cast<uint32_t>(before >> 32);
    uint32_t eq_seen = static_cast<uint32_t>(before & 0xFFFFFFFFu);
    uint32_t pos = gt_before + min(eq_seen, krem);
    for_keys([&](int i, uint32_t key) {
        const uint32_t km = key & pmask;
        if (km > kstar || (km == kstar && eq_seen++ < krem))
            out[pos++] = idx_base + static_cast<int>(i0) + i;
    });
    if (C > 1) cluster_wait();   // others may still read this CTA's counts until here
}

// ---- one CTA, up to kSmallN keys -------------------------------------------------
//
// For small inputs the cluster machinery costs more than the counting, so one CTA of
// kNT threads (8 or 16 keys each, in registers) runs a leaner form of the same exact
// selection:
//   - the digits start at the highest bit in which the smallest and largest key differ
//     (every key shares the bits above it), so the first 11-bit digit already splits
//     the populated key range;
//   - after each histogram one warp finds the bin of the k-th largest key: lane l sums
//     the 64 bins [2048 - 64(l+1), 2048 - 64 l) (lane 0 the highest), a warp scan picks
//     the lane, a second scan over that lane's bins (two per lane) picks the bin; the
//     rest of the CTA waits at one barrier;
//   - when that bin holds at most kCand keys and not all of them are taken, its keys are
//     gathered in shared memory and one warp ranks them directly (each candidate counts
//     the candidates above it), which gives K* without further passes;
//   - the final counts (greater, equal) fit in 16 bits each, so one 32-bit block scan
//     gives every thread its first output position.
constexpr int kSmallN = kNT * 16;
constexpr int kCand = 64;

struct SmallShared {
    uint32_t hist[2][kBins];            // double-buffered: a pass clears the one it read
    uint32_t wmin[kWarps], wmax[kWarps];
    uint32_t wsum[kWarps];
    uint32_t cand[kCand];
    uint32_t s_hit, s_above, s_cnt, s_ncand, s_kstar, s_krem;
};

// Warp 0 only: the bin of hist (kBins bins, digit order) that holds the krem-th largest
// key, the keys above it and its count, into s_hit / s_above / s_cnt.  The histogram
// holds at least krem keys.
__device__ __forceinline__ void small_find_bin(const uint32_t *hist, uint32_t krem,
                                               SmallShared *s) {
    const int lane = threadIdx.x & 31;
    const uint4 *h4 = reinterpret_cast<const uint4 *>(hist) + (kBins - 64 * (lane + 1)) / 4;
    uint32_t sum = 0;
#pragma unroll
    for (int q = 0; q < 16; ++q) {   // rotated start: the lanes of a phase hit distinct banks
        const uint4 v = h4[(q + lane) & 15];
        sum += v.x + v.y + v.z + v.w;
    }
    const uint32_t incl = warp_incl_scan(sum);
    const uint32_t above = incl - sum;
    const int L = __ffs(__ballot_sync(0xFFFFFFFFu, above < krem && incl >= krem)) - 1;
    const uint32_t above_l = __shfl_sync(0xFFFFFFFFu, above, L);
    // lane j: bins b and b - 1 of lane L's chunk, b = its top bin - 2j (descending)
    const int b = kBins - 64 * L - 1 - 2 * lane;
    const uint32_t f1 = hist[b], f2 = hist[b - 1];
    const uint32_t incl2 = warp_incl_scan(f1 + f2);
    const uint32_t above2 = incl2 - f1 - f2, want = krem - above_l;
    if (above2 < want && incl2 >= want) {
        const bool top = above2 + f1 >= want;
        s->s_hit = static_cast<uint32_t>(top ? b : b - 1);
        s->s_above = above_l + (top ? above2 : above2 + f1);
        s->s_cnt = top ? f1 : f2;
    }
}

template <int KPT>
__global__ void __launch_bounds__(kNT, 1)
select_small_kernel(const uint32_t *__restrict__ score, int n, int k, int idx_base, int vec,
                    int *__restrict__ out) {
    pdl_wait();   // inputs may come from the previous kernel of the stream
    pdl_trigger();
    __shared__ __align__(16) SmallShared sh;
    SmallShared *s = &sh;
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    const int i0 = t * KPT;
    const int cnt = max(0, min(KPT, n - i0));
    if (k >= n) {   // everything is selected, in index order (no barrier on this path)
        for (int i = 0; i < cnt; ++i) out[i0 + i] = idx_base + i0 + i;
        return;
    }
    uint32_t reg[KPT];
    if (vec && cnt == KPT) {
#pragma unroll
        for (int c = 0; c < KPT / 4; ++c) {
            const uint4 u = __ldg(reinterpret_cast<const uint4 *>(score + i0) + c);
            reg[4 * c] = order_key(u.x);
            reg[4 * c + 1] = order_key(u.y);
            reg[4 * c + 2] = order_key(u.z);
            reg[4 * c + 3] = order_key(u.w);
        }
    } else {
#pragma unroll
        for (int i = 0; i < KPT; ++i) reg[i] = i < cnt ? order_key(__ldg(score + i0 + i)) : 0u;
    }
    uint32_t lo = 0xFFFFFFFFu, hi = 0u;
#pragma unroll
    for (int i = 0; i < KPT; ++i)
        if (i < cnt) {
            lo = min(lo, reg[i]);
            hi = max(hi, reg[i]);
        }
    lo = __reduce_min_sync(0xFFFFFFFFu, lo);
    hi = __reduce_max_sync(0xFFFFFFFFu, hi);
    if (lane == 0) {
        s->wmin[warp] = lo;
        s->wmax[warp] = hi;
    }
    {
        uint4 *h = reinterpret_cast<uint4 *>(&s->hist[0][0]);
        for (int j = t; j < 2 * kBins / 4; j += kNT) h[j] = make_uint4(0, 0, 0, 0);
    }
    if (t == 0) {
        s->s_ncand = 0;
        s->s_hit = 0;
        s->s_above = 0;
        s->s_cnt = 0;
        s->s_kstar = 0;
        s->s_krem = 0;
    }
    __syncthreads();
    const uint32_t kmin = __reduce_min_sync(0xFFFFFFFFu, s->wmin[lane % kWarps]);
    const uint32_t kmax = __reduce_max_sync(0xFFFFFFFFu, s->wmax[lane % kWarps]);

    // prefix = the resolved high bits of K*, pmask their mask; krem = how many keys with
    // that prefix are still to be selected; nxt = the number of unresolved low bits
    const uint32_t diff = kmin ^ kmax;
    int nxt = diff ? 32 - __clz(diff) : 0;
    uint32_t pmask = nxt == 32 ? 0u : ~((1u << nxt) - 1u);
    uint32_t prefix = kmax & pmask;
    uint32_t krem = static_cast<uint32_t>(k);
    int buf = 0;
#pragma unroll 1
    while (nxt > 0) {
        const int shift = max(nxt - 11, 0);
        const uint32_t dmask = (1u << (nxt - shift)) - 1u;
        uint32_t *hist = s->hist[buf];
#pragma unroll
        for (int i = 0; i < KPT; ++i)
            if (i < cnt && (reg[i] & pmask) == prefix) atomicAdd(&hist[(reg[i] >> shift) & dmask], 1u);
        __syncthreads();
        if (warp == 0) small_find_bin(hist, krem, s);
        __syncthreads();
        const uint32_t c_bin = s->s_cnt;
        prefix |= s->s_hit << shift;
        pmask |= dmask << shift;
        krem -= s->s_above;
        nxt = shift;
        // every key left in the bin is taken, or the bin is one key value: K* is resolved
        // as far as the selection needs
        if (c_bin == krem || nxt == 0) break;
        if (c_bin <= static_cast<uint32_t>(kCand)) {
            // rank the bin's keys directly
#pragma unroll
            for (int i = 0; i < KPT; ++i)
                if (i < cnt && (reg[i] & pmask) == prefix) s->cand[atomicAdd(&s->s_ncand, 1u)] = reg[i];
            __syncthreads();
            if (warp == 0) {
                for (int j = lane; j < static_cast<int>(c_bin); j += 32) {
                    const uint32_t x = s->cand[j];
                    uint32_t gt = 0, ge = 0;
                    for (int q = 0; q < static_cast<int>(c_bin); ++q) {
                        const uint32_t y = s->cand[q];
                        gt += y > x;
                        ge += y >= x;
                    }
                    if (gt < krem && ge >= krem) {   // x is K* (equal candidates agree)
                        s->s_kstar = x;
                        s->s_krem = krem - gt;
                    }
                }
            }
            __syncthreads();
            prefix = s->s_kstar;
            pmask = 0xFFFFFFFFu;
            krem = s->s_krem;
            break;
        }
        // another histogram pass over the next digit: clear the buffer just read (the
        // pass after next uses it; a barrier separates the two)
        for (int j = t; j < kBins / 4; j += kNT)
            reinterpret_cast<uint4 *>(hist)[j] = make_uint4(0, 0, 0, 0);
        buf ^= 1;
    }

    // K* = prefix under pmask; keys above it are taken, and the first krem equal to it
    const uint32_t kstar = prefix;
    uint32_t gt = 0, eq = 0;
#pragma unroll
    for (int i = 0; i < KPT; ++i)
        if (i < cnt) {
            const uint32_t km = reg[i] & pmask;
            gt += km > kstar;
            eq += km == kstar;
        }
    // both counts stay below 2^16 over the whole CTA (n <= kSmallN)
    const uint32_t mine = (gt << 16) | eq;
    const uint32_t before = block_incl_scan<uint32_t>(mine, s->wsum) - mine;
    uint32_t eq_seen = before & 0xFFFFu;
    uint32_t pos = (before >> 16) + min(eq_seen, krem);
#pragma unroll
    for (int i = 0; i < KPT; ++i)
        if (i < cnt) {
            const uint32_t km = reg[i] & pmask;
            if (km > kstar || (km == kstar && eq_seen++ < krem)) out[pos++] = idx_base + i0 + i;
        }
}

// The largest cluster size (a power of two <= 16) the device can co-schedule for
// kernel number `which` (0..3); cached per kernel and device.
int max_cluster(int which, void (*kernel)(const uint32_t *, int, int, int, int, int, int *)) {
    static std::mutex mu;
    static int cached[4][64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
    std::lock_guard<std::mutex> lock(mu);
    int &slot = cached[which][dev];
    if (slot == 0) {
        int best = 1;
        if (cudaFuncSetAttribute(kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
            cudaSuccess)
            (void)cudaGetLastError();
        for (int c = kMaxCluster; c >= 2; c /= 2) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(c);
            cfg.blockDim = dim3(kNT);
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeClusterDimension;
            attr[0].val.clusterDim.x = c;
            attr[0].val.clusterDim.y = 1;
            attr[0].val.clusterDim.z = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            int nclusters = 0;
            if (cudaOccupancyMaxActiveClusters(&nclusters, kernel, &cfg) == cudaSuccess &&
                nclusters >= 1) {
                best = c;
                break;
            }
            (void)cudaGetLastError();
        }
        slot = best;
    }
    return slot;
}

template <int KPT>
cudaError_t launch_kpt(int C, const uint32_t *keys, int n, int k, int idx_base, int per, int vec,
                       int *out, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(C);
    cfg.blockDim = dim3(kNT);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    int na = 0;
    attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[na].val.programmaticStreamSerializationAllowed = 1;
    ++na;
    if (C > 1) {
        attr[na].id = cudaLaunchAttributeClusterDimension;
        attr[na].val.clusterDim.x = C;
        attr[na].val.clusterDim.y = 1;
        attr[na].val.clusterDim.z = 1;
        ++na;
    }
    cfg.attrs = attr;
    cfg.numAttrs = na;
    return cudaLaunchKernelEx(&cfg, select_kernel<KPT>, keys, n, k, idx_base, per, vec, out);
}

}  // namespace

cudaError_t launch_select(const float *score, int n, int k, int idx_base, int *out,
                          cudaStream_t s) {
    if (k == 0 || n == 0) return cudaSuccess;
    const uint32_t *keys = reinterpret_cast<const uint32_t *>(score);
    const int vec = (reinterpret_cast<uintptr_t>(score) & 15u) == 0;
    if (n <= kSmallN) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(1);
        cfg.blockDim = dim3(kNT);
        cfg.stream = s;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (n <= kNT * 8)
            return cudaLaunchKernelEx(&cfg, select_small_kernel<8>, keys, n, k, idx_base, vec, out);
        return cudaLaunchKernelEx(&cfg, select_small_kernel<16>, keys, n, k, idx_base, vec, out);
    }
    // cluster size: about 4096 keys per CTA, a power of two up to what the device allows
    int want = 1;
    while (want < kMaxCluster && static_cast<long long>(want) * 4096 < n) want *= 2;
    // every variant must be able to run the cluster (the choice of variant below depends on C)
    int cap = max_cluster(0, select_kernel<4>);
    cap = std::min(cap, max_cluster(1, select_kernel<8>));
    cap = std::min(cap, max_cluster(2, select_kernel<16>));
    cap = std::min(cap, max_cluster(3, select_kernel<0>));
    const int C = std::min(want, cap);
    // keys per thread for that cluster: in registers up to 16, else re-read per pass
    const long long per_thread = (n + static_cast<long long>(C) * kNT - 1) / (static_cast<long long>(C) * kNT);
    if (per_thread <= 4) return launch_kpt<4>(C, keys, n, k, idx_base, 4, vec, out, s);
    if (per_thread <= 8) return launch_kpt<8>(C, keys, n, k, idx_base, 8, vec, out, s);
    if (per_thread <= 16) return launch_kpt<16>(C, keys, n, k, idx_base, 16, vec, out, s);
    const int per = static_cast<int>((per_thread + 3) / 4 * 4);
    return launch_kpt<0>(C, keys, n, k, idx_base, per, vec, out, s);
}

}  // namespace cs
