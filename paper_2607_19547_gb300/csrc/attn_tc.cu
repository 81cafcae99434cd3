// Step 4 for bf16 storage: repair attention on the fifth-generation tensor
// cores (ChronoStitch Eq. 1 over the selected rows, causal in global sequence
// order, Sec. 2).
//
// Work tile: (layer l, kv head g, query tile).  A query tile packs the G
// query heads that share kv head g for TOK = 128/G consecutive selected rows
// into one 128-row MMA operand (row m = token*G + head), so every K/V tile
// loaded from HBM feeds all G heads.  The tile walks key blocks of 128 up to
// the largest qpos of its rows; blocks past the smallest qpos apply the
// per-row causal mask.
//
// CTA = 11 warps:
//   warp 0      TMA producers: lane 0 loads Q once and streams K through a
//               3-stage shared-memory ring, lane 1 streams V through a
//               2-stage ring (128-byte swizzle).
//   warp 1      owns tensor memory; lane 0 issues S_j = Q K_j^T (A, B from
//               shared memory, fp32 into one of three 128-column TMEM buffers).
//   warp 10     lane 0 issues O += P_j V_j (A = P_j from TMEM, B = V from
//               shared memory, MN-major).
//               A tcgen05.mma issue blocks until the tensor core takes it, so
//               one thread that also waits on barriers leaves the tensor core
//               idle while it waits; two issuers keep it fed.
//   warps 2-9   softmax, two warpgroups: warpgroup h (warps 2+4h .. 5+4h)
//               owns key columns [64h, 64h+64) of every S block and output
//               dims [64h, 64h+64) of O; thread = one TMEM lane = one query
//               row.  Reads its half of S_j, masks it and computes its half of
//               P_j = exp2(...) with the running max of the earlier blocks; the
//               sum of those weights flags a block that may hold a larger
//               maximum (above 2^12, or not finite).  It then meets the warp
//               that holds the other half of the same 32 rows (a 64-thread
//               named barrier with an OR per block; the four row quarters run
//               independently).  When either half flagged (and on the first
//               block), both warps take their half-row maxima of S_j, exchange
//               them through shared memory, raise the running max if it grew by
//               more than 2^8, recompute P_j from S_j and rescale their half of
//               O in TMEM.  Each warp writes
//               its half of P_j as bf16 over the first 32 of its own 64 S_j
//               columns (never over columns the other warp reads), and the P*V
//               issuer takes keys [64h, 64h+64) from columns [64h, 64h+32).
//               Finally each warp normalises
//               its half of O into the Q tile's shared memory (idle after the
//               last S), from where two TMA stores write whole rows.
// TMEM: S buffers at columns 0, 128, 256; O at 384.  S_j reuses the buffer
// of P_{j-3}, so the S issuer runs up to three blocks ahead of the softmax.
// Every mbarrier wait is bounded; on a timeout the CTA records
// CS_ERR_TIMEOUT, stops issuing work, drains what it issued, frees its
// tensor memory and exits.
#include <cuda.h>

#include <algorithm>
#include <mutex>

#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kThreads = 352;          // 11 warps: producers, S issuer, 2 x 4 softmax, PV issuer
constexpr int kPvWarp = 10;
constexpr int kBlockN = 128;           // keys per KV block
constexpr int kKStages = 3;            // K shared-memory ring depth
constexpr int kVStages = 2;            // V ring depth (V is consumed after the softmax)
constexpr uint32_t kHalf = 128 * 64 * 2;           // 128 rows x 64 dims (one swizzle half)
constexpr uint32_t kTileBytes = 2 * kHalf;         // Q tile, or one K or V block
constexpr uint32_t kTmemCols = 512;
constexpr int kSBufs = 3;              // S (and P) buffers of 128 columns
constexpr uint32_t kColO = 384;
constexpr uint64_t kWaitLimitNs = 1000000000ull;    // 1 s

struct Smem {
    // byte offsets from the 1024-aligned base
    static constexpr uint32_t q = 0;
    static constexpr uint32_t k = q + kTileBytes;
    static constexpr uint32_t v = k + kKStages * kTileBytes;
    static constexpr uint32_t bars = v + kVStages * kTileBytes;
    static constexpr uint32_t xchg = bars + 512;           // float [2 slots][2 halves][128 rows]
    static constexpr uint32_t total = xchg + 2 * 2 * 128 * 4;
};

struct Bars {
    uint64_t q_full;
    uint64_t k_full[kKStages], k_empty[kKStages];
    uint64_t v_full[kVStages], v_empty[kVStages];
    uint64_t s_full[kSBufs], p_full[kSBufs];
    uint64_t pv_done[kSBufs];   // one completion per P*V block that read P from buffer b
    uint64_t o_final;           // single use: every P*V of the tile is done
    uint64_t mma_done;          // single use (two arrivals): every tensor-core operation retired
    uint32_t tmem_base;
    int abort;
};
static_assert(sizeof(Bars) <= 512, "barrier area");

struct TcParams {
    int n_layers, M, T, hq, hkv, G, tok, n_qtiles;
    float scale_log2;
    float *lse;
    __nv_bfloat16 *o;
    const int *qpos;
    unsigned int *status;
};

__device__ __forceinline__ uint32_t ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return __float_as_uint(y);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// One warp's 64-column half of an S block from TMEM (its lane = its row), with the
// causal mask applied on blocks that reach past the row's position: columns above
// `lim` become -inf.
__device__ __forceinline__ void load_s_half(uint32_t taddr, bool diag, int lim, float (&s)[64]) {
    uint32_t sr[64];
    tmem_ld64(taddr, sr);
#pragma unroll
    for (int c = 0; c < 64; ++c) s[c] = __uint_as_float(sr[c]);
    if (diag) {
#pragma unroll
        for (int c = 0; c < 64; ++c)
            if (c > lim) s[c] = -INFINITY;
    }
}

// P = exp2(s * scale * log2(e) - m) for 64 columns, packed as bf16 pairs; returns the
// fp32 sum of the 64 weights (affine step and sum in fp32x2).
__device__ __forceinline__ float exp_pack(const float (&s)[64], float scale_log2, float m,
                                          uint32_t (&pk)[32]) {
    const float2 sc2 = make_float2(scale_log2, scale_log2);
    const float2 nm2 = make_float2(-m, -m);
    float2 psum = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int e = 0; e < 32; ++e) {
        const float2 tt = __ffma2_rn(make_float2(s[2 * e], s[2 * e + 1]), sc2, nm2);
        const float2 pe = make_float2(__uint_as_float(ex2_approx(tt.x)),
                                      __uint_as_float(ex2_approx(tt.y)));
        psum = __fadd2_rn(psum, pe);
        pk[e] = pack_bf16x2(pe.x, pe.y);
    }
    return psum.x + psum.y;
}

// Tile coordinates of work item `item`.  CTAs launched together should share
// a (layer, kv head) so its K/V blocks are read from HBM once and then hit in
// L2; to keep the tail short the heavier half of the query tiles (selected
// rows ascend, so later tiles see more keys) runs first for every group, then
// the lighter half.  Within a group, tiles run heaviest first.
__device__ __forceinline__ void decode_item(const TcParams &p, int item, int &l, int &g, int &qt) {
    const int lo_n = p.n_qtiles / 2, hi_n = p.n_qtiles - lo_n;
    const int groups = p.n_layers * p.hkv;
    int grp;
    if (item < groups * hi_n) {
        grp = item / hi_n;
        qt = p.n_qtiles - 1 - item % hi_n;
    } else {
        const int i2 = item - groups * hi_n;
        grp = i2 / lo_n;
        qt = lo_n - 1 - i2 % lo_n;
    }
    l = grp / p.hkv;
    g = grp % p.hkv;
}

__device__ __forceinline__ int clamp_pos(int x, int T) { return min(max(x, 0), T - 1); }

__global__ void __launch_bounds__(kThreads, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
               const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_o,
               const TcParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    Bars *bars = reinterpret_cast<Bars *>(base + Smem::bars);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    int l, g, qt;
    decode_item(p, blockIdx.x, l, g, qt);
    const int r0 = qt * p.tok;
    const int r_last = min(p.M, r0 + p.tok) - 1;
    const uint32_t q_bytes = static_cast<uint32_t>(p.tok * p.G) * 256u;   // both 64-column halves

    if (warp == 0) {
        // thread 0 is the Q/K producer: Q and the first K block go out before the other
        // barriers are initialised and before the CTA-wide barrier (nothing else
        // touches these barriers until after it); lanes initialise the rest in parallel
        if (lane == 0) {
            mbar_init(&bars->q_full, 1);
            mbar_init(&bars->k_full[0], 1);
            fence_mbar_init();
            tma_prefetch_desc(&tm_q);
            tma_prefetch_desc(&tm_k);
            mbar_arrive_expect_tx(&bars->q_full, q_bytes);
            tma_load_4d(base + Smem::q, &tm_q, &bars->q_full, 0, g * p.G, r0, l);
            tma_load_4d(base + Smem::q + kHalf, &tm_q, &bars->q_full, 64, g * p.G, r0, l);
            mbar_arrive_expect_tx(&bars->k_full[0], kTileBytes);
            tma_load_4d(base + Smem::k, &tm_k, &bars->k_full[0], 0, g, 0, l);
            tma_load_4d(base + Smem::k + kHalf, &tm_k, &bars->k_full[0], 64, g, 0, l);
        }
        if (lane >= 1 && lane < kKStages) mbar_init(&bars->k_full[lane], 1);
        if (lane < kKStages) mbar_init(&bars->k_empty[lane], 1);
        if (lane < kVStages) {
            mbar_init(&bars->v_full[lane], 1);
            mbar_init(&bars->v_empty[lane], 1);
        }
        if (lane < kSBufs) {
            mbar_init(&bars->s_full[lane], 1);
            mbar_init(&bars->p_full[lane], 256);
            mbar_init(&bars->pv_done[lane], 1);
        }
        if (lane == 8) mbar_init(&bars->o_final, 1);
        if (lane == 9) mbar_init(&bars->mma_done, 2);
        if (lane == 10) bars->abort = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&bars->tmem_base, kTmemCols);
        tmem_relinquish();
    }
    // rows of the Q tile that TMA does not write (G not dividing 128) must be finite
    {
        const uint32_t used = static_cast<uint32_t>(p.tok * p.G) * 128u;   // bytes per half
        for (uint32_t off = used + threadIdx.x * 16u; off < kHalf; off += kThreads * 16u) {
            *reinterpret_cast<uint4 *>(base + Smem::q + off) = make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4 *>(base + Smem::q + kHalf + off) = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async_smem();
    }
    // the positions are read only now: a release fence above (the barrier-init fence)
    // would otherwise wait for these global loads before the Q and K copies go out
    const int qmin = clamp_pos(p.qpos[r0], p.T);
    const int kmax = clamp_pos(p.qpos[r_last], p.T);
    const int nb = kmax / kBlockN + 1;
    const int mask_from = qmin / kBlockN;
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int *abort = &bars->abort;

    if (warp == 0) {
        // ------------------------------------------------------------ producers
        // lane 0 streams the K ring (Q and K block 0 went out at set-up), lane 1 the V ring
        if (lane < 2) {
            volatile int never = 0;
            int issued = lane == 0 ? 1 : 0;
            const int stages = lane == 0 ? kKStages : kVStages;
            uint64_t *full = lane == 0 ? bars->k_full : bars->v_full;
            uint64_t *empty = lane == 0 ? bars->k_empty : bars->v_empty;
            const CUtensorMap *tm = lane == 0 ? &tm_k : &tm_v;
            const uint32_t ring = lane == 0 ? Smem::k : Smem::v;
            if (lane == 1) tma_prefetch_desc(tm);
            for (int j = issued; j < nb; ++j) {
                const int s = j % stages;
                if (!mbar_wait_bounded(&empty[s], ((j / stages) & 1) ^ 1, abort, p.status,
                                       kSiteAttnProducer, kWaitLimitNs)) break;
                uint8_t *dst = base + ring + s * kTileBytes;
                mbar_arrive_expect_tx(&full[s], kTileBytes);
                tma_load_4d(dst, tm, &full[s], 0, g, j * kBlockN, l);
                tma_load_4d(dst + kHalf, tm, &full[s], 64, g, j * kBlockN, l);
                ++issued;
            }
            if (*abort) {
                // drain: every issued copy lands before the CTA's shared memory is released.
                // Phases of one barrier complete in order, so waiting for the last copy
                // issued on each barrier covers the earlier ones.
                if (lane == 0) mbar_wait_bounded(&bars->q_full, 0, &never, nullptr, 0, kWaitLimitNs);
                for (int s = 0; s < stages; ++s) {
                    if (issued <= s) continue;
                    const int jl = s + ((issued - 1 - s) / stages) * stages;
                    mbar_wait_bounded(&full[s], (jl / stages) & 1, &never, nullptr, 0, kWaitLimitNs);
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ S issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(128, kBlockN, 0, 0);
            // descriptors are built once; an operand at byte offset `off` from a base is
            // base + (off >> 4) (the 14-bit address field cannot overflow below 256 KB)
            const uint64_t qd = smem_desc(smem_u32(base + Smem::q), 16, 1024, 2);
            const uint64_t kd0 = smem_desc(smem_u32(base + Smem::k), 16, 1024, 2);
            bool ok = mbar_wait_bounded(&bars->q_full, 0, abort, p.status, kSiteAttnMma,
                                        kWaitLimitNs);
            for (int j = 0; ok && j < nb; ++j) {
                const int s = j % kKStages, b = j % kSBufs;
                // buffer b held P_{j-3}: PV_{j-3} must have read it
                if (j >= kSBufs && !mbar_wait_bounded(&bars->pv_done[b], ((j / kSBufs) - 1) & 1,
                                                      abort, p.status, kSiteAttnMma, kWaitLimitNs)) break;
                if (!mbar_wait_bounded(&bars->k_full[s], (j / kKStages) & 1, abort, p.status,
                                       kSiteAttnMma, kWaitLimitNs)) break;
                tc_fence_after();
                const uint64_t kd = kd0 + ((s * kTileBytes) >> 4);
                const uint32_t d = tmem + static_cast<uint32_t>(b * kBlockN);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {   // 16 head dims per MMA
                    const uint32_t off = (kk >> 2) * kHalf + (kk & 3) * 32;
                    tc_mma_ss(d, qd + (off >> 4), kd + (off >> 4), idesc, kk > 0);
                }
                tc_commit(&bars->s_full[b]);
                tc_commit(&bars->k_empty[s]);
            }
            // completes once every tcgen05 operation issued by this thread has retired
            tc_commit(&bars->mma_done);
        }
    } else if (warp == kPvWarp) {
        // ------------------------------------------------------------ PV issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16(128, 128, 0, 1);
            const uint64_t vd0 = smem_desc(smem_u32(base + Smem::v), kHalf, 1024, 2);
            for (int j = 0; j < nb; ++j) {
                const int s = j % kVStages, b = j % kSBufs;
                if (!mbar_wait_bounded(&bars->p_full[b], (j / kSBufs) & 1, abort, p.status,
                                       kSiteAttnMma, kWaitLimitNs)) break;
                if (!mbar_wait_bounded(&bars->v_full[s], (j / kVStages) & 1, abort, p.status,
                                       kSiteAttnMma, kWaitLimitNs)) break;
                tc_fence_after();
                const uint64_t vd = vd0 + ((s * kTileBytes) >> 4);
                const uint32_t a_tm = tmem + static_cast<uint32_t>(b * kBlockN);
#pragma unroll
                for (int kk = 0; kk < kBlockN / 16; ++kk) {
                    // A: 16 keys of P = 8 packed columns (keys [64h, 64h+64) sit in columns
                    // [64h, 64h+32) of the buffer); B: 16 rows (keys) of V, MN-major
                    tc_mma_ts(tmem + kColO, a_tm + (kk >> 2) * 64 + (kk & 3) * 8,
                              vd + ((kk * 2048) >> 4), idesc, (j > 0 || kk > 0) ? 1u : 0u);
                }
                tc_commit(&bars->pv_done[b]);
                tc_commit(&bars->v_empty[s]);
                if (j == nb - 1) tc_commit(&bars->o_final);
            }
            tc_commit(&bars->mma_done);
        }
    } else {
        // ------------------------------------------------------------ softmax
        const int half = (warp - 2) >> 2;             // key columns / output dims [64h, 64h+64)
        const int qw = warp & 3;
        const int m = 32 * qw + lane;                 // TMEM lane = MMA row
        const int t = m / p.G, hh = m - t * p.G;
        const int r = r0 + t;
        const bool valid = (m < p.tok * p.G) && (r <= r_last);
        int qp = kmax;
        if (valid) {
            const int raw = p.qpos[r];
            if (half == 0 && (raw < 0 || raw >= p.T || (r > 0 && p.qpos[r - 1] >= raw)))
                report_error(p.status, 5u, kSiteAttnQpos, static_cast<unsigned>(r));
            qp = clamp_pos(raw, p.T);
        }
        float *xchg = reinterpret_cast<float *>(base + Smem::xchg);   // [slot][half][row]
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * qw) << 16);
        const int col0 = 64 * half;
        float m_run = -INFINITY, l_run = 0.0f;
        bool ok = true;
        // Failure handling: a thread that gives up only clears `ok`; the decision to
        // stop is taken by both warps of a row quarter together at their exchange
        // barrier (barrier + OR), so neither is ever left waiting there; a quarter that
        // stops raises `abort`, which ends the other quarters' bounded waits, and every
        // softmax thread then meets the others at the epilogue's barriers.
        for (int j = 0; j < nb; ++j) {
            const int b = j % kSBufs;
            if (ok) {
                const bool w_ok = mbar_wait_bounded(&bars->s_full[b], (j / kSBufs) & 1, abort,
                                                    p.status, kSiteAttnSoftmax, kWaitLimitNs);
                ok = __all_sync(0xFFFFFFFFu, w_ok);
            }
            float *slot = xchg + (j & 1) * 256;
            const uint32_t s_addr = lane_base + b * kBlockN + col0;
            const bool diag = j >= mask_from;
            const int lim = qp - j * kBlockN - col0;
            float psum = 0.0f;
            uint32_t pk[32];
            bool grow = true;   // the first block always sets the running max
            if (ok && j > 0) {
                // this half of P_j with the running max of the earlier blocks; the sum of
                // the weights flags a block that may hold a larger maximum (it exceeds 2^12,
                // or is not finite), and only then do the warps take the half maxima (below)
                tc_fence_after();
                float s[64];
                load_s_half(s_addr, diag, lim, s);
                psum = exp_pack(s, p.scale_log2, m_run, pk);
                grow = !(psum <= 4096.0f);
            }
            // the two warps that own a row's halves (same TMEM lane quarter) meet here;
            // the four pairs run independently of one another.  A failure or a flagged
            // block in either warp takes both through the exchange of the half maxima.
            bool rescale = false;
            float alpha = 1.0f;
            if (named_bar_red_or(2 + qw, 64, !ok || grow)) {
                if (named_bar_red_or(2 + qw, 64, !ok)) {
                    ok = false;
                    *abort = 1;
                    break;
                }
                // S_j is still in TMEM (P_j has not been written over it yet)
                float s[64];
                tc_fence_after();
                load_s_half(s_addr, diag, lim, s);
                {
                    float mx4[4] = {s[0], s[1], s[2], s[3]};
#pragma unroll
                    for (int c = 4; c < 64; c += 4) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) mx4[q] = fmaxf(mx4[q], s[c + q]);
                    }
                    slot[half * 128 + m] = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
                }
                named_bar_sync(2 + qw, 64);   // both halves' maxima are in the slot
                const float mx2 = fmaxf(slot[m], slot[128 + m]) * p.scale_log2;
                const bool g = (m_run == -INFINITY) || (mx2 > m_run + 8.0f);
                if (g) {
                    alpha = exp2f(m_run - mx2);   // 0 on the first block
                    l_run *= alpha;
                    m_run = mx2;
                }
                rescale = j > 0 && __any_sync(0xFFFFFFFFu, g);
                psum = exp_pack(s, p.scale_log2, m_run, pk);
            }
            // packed bf16 into columns [64h, 64h+32) of S_j's buffer: inside this warp's
            // own half of S_j, which it has read already, so no other warp's read of S_j can
            // meet this store
            tmem_st32(lane_base + b * kBlockN + col0, pk);
            l_run += psum;
            // rescale this half of O when any row of the warp raised its max
            // (O holds PV_0 .. PV_{j-1})
            if (rescale) {
                const bool o_ok = mbar_wait_bounded(&bars->pv_done[(j - 1) % kSBufs],
                                                    ((j - 1) / kSBufs) & 1, abort, p.status,
                                                    kSiteAttnSoftmax, kWaitLimitNs);
                ok = __all_sync(0xFFFFFFFFu, o_ok);
                if (ok) {
                    tc_fence_after();
                    uint32_t orr[64];
                    tmem_ld64(lane_base + kColO + col0, orr);
#pragma unroll
                    for (int e = 0; e < 64; ++e)
                        orr[e] = __float_as_uint(__uint_as_float(orr[e]) * alpha);
                    tmem_st64(lane_base + kColO + col0, orr);
                }
            }
            tc_fence_before();
            mbar_arrive(&bars->p_full[b]);
        }
        if (ok) {
            const bool w_ok = mbar_wait_bounded(&bars->o_final, 0, abort, p.status,
                                                kSiteAttnSoftmax, kWaitLimitNs);
            ok = __all_sync(0xFFFFFFFFu, w_ok);
        }
        // combine the two halves' row sums (slot 0 of the exchange array; every
        // thread has passed its last read of it)
        named_bar_sync(1, 256);
        xchg[half * 128 + m] = l_run;
        const bool fail = named_bar_red_or(1, 256, !ok || *abort);
        const float l_tot = xchg[m] + xchg[128 + m];
        if (!fail) {
            tc_fence_after();
            const float inv = 1.0f / l_tot;
            uint32_t orr[64];
            tmem_ld64(lane_base + kColO + col0, orr);
            // O leaves through shared memory: the Q tile (no MMA reads it after the last
            // S) in the same 128-byte-swizzled layout, then one TMA store per half, so
            // the global writes are whole rows; rows past M are clipped by the store
            uint8_t *orow = base + Smem::q + half * kHalf + m * 128;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                uint32_t w4[4];
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    w4[q] = pack_bf16x2(__uint_as_float(orr[8 * e + 2 * q]) * inv,
                                        __uint_as_float(orr[8 * e + 2 * q + 1]) * inv);
                *reinterpret_cast<uint4 *>(orow + ((e ^ (m & 7)) << 4)) =
                    make_uint4(w4[0], w4[1], w4[2], w4[3]);
            }
            if (valid && half == 0 && p.lse != nullptr)
                p.lse[(static_cast<long long>(l) * p.M + r) * p.hq + g * p.G + hh] =
                    (m_run + __log2f(l_tot)) * 0.69314718055994531f;
            fence_proxy_async_smem();
        }
        named_bar_sync(1, 256);   // `fail` is the same in every softmax thread
        if (!fail && threadIdx.x == 64) {
            tma_store_4d(&tm_o, base + Smem::q, 0, g * p.G, r0, l);
            tma_store_4d(&tm_o, base + Smem::q + kHalf, 64, g * p.G, r0, l);
            bulk_commit();
            bulk_wait_read();   // the stores have read shared memory before the CTA exits
        }
    }
    // tensor memory is released only after every tensor-core operation retired
    if (warp == 1 && lane == 0) {
        volatile int never = 0;
        mbar_wait_bounded(&bars->mma_done, 0, &never, nullptr, 0, kWaitLimitNs);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

// ---- host side --------------------------------------------------------------

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                   const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                   const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    });
    return fn;
}

bool make_map(EncodeTiledFn enc, CUtensorMap *map, const void *ptr, const cuuint64_t dims[4],
              const cuuint64_t strides[3], const cuuint32_t box[4]) {
    const cuuint32_t elem_strides[4] = {1, 1, 1, 1};
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(ptr), dims, strides,
               box, elem_strides, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

}  // namespace

cs_status launch_attn_tc(const AttnArgs &a, cudaStream_t s) {
    const int G = a.hq / a.hkv;
    const int tok = 128 / G;
    const int n_qtiles = (a.M + tok - 1) / tok;
    const long long items = static_cast<long long>(n_qtiles) * a.n_layers * a.hkv;
    if (items == 0) return CS_OK;
    if (items > 0x7FFFFFFFll) return fail(CS_ERR_UNSUPPORTED, "too many attention tiles");
    EncodeTiledFn enc = get_encode_fn();
    if (enc == nullptr) return fail(CS_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
    CUtensorMap tq, tk, tv, to;
    const cuuint64_t qdims[4] = {128, static_cast<cuuint64_t>(a.hq), static_cast<cuuint64_t>(a.M),
                                 static_cast<cuuint64_t>(a.n_layers)};
    const cuuint64_t qstr[3] = {256ull, 256ull * a.hq, 256ull * a.hq * a.M};
    const cuuint32_t qbox[4] = {64, static_cast<cuuint32_t>(G), static_cast<cuuint32_t>(tok), 1};
    const cuuint64_t kdims[4] = {128, static_cast<cuuint64_t>(a.hkv), static_cast<cuuint64_t>(a.T),
                                 static_cast<cuuint64_t>(a.n_layers)};
    const cuuint64_t kstr[3] = {256ull, 256ull * a.hkv, 2ull * static_cast<cuuint64_t>(a.kv_layer_stride)};
    const cuuint32_t kbox[4] = {64, 1, static_cast<cuuint32_t>(kBlockN), 1};
    if (!make_map(enc, &tq, a.q, qdims, qstr, qbox) || !make_map(enc, &to, a.o, qdims, qstr, qbox) ||
        !make_map(enc, &tk, a.k, kdims, kstr, kbox) ||
        !make_map(enc, &tv, a.v, kdims, kstr, kbox))
        return fail(CS_ERR_INVALID_ARG, "tensor map encoding failed (alignment or extent)");
    TcParams p;
    p.n_layers = a.n_layers;
    p.M = a.M;
    p.T = a.T;
    p.hq = a.hq;
    p.hkv = a.hkv;
    p.G = G;
    p.tok = tok;
    p.n_qtiles = n_qtiles;
    p.scale_log2 = a.scale * 1.4426950408889634f;
    p.lse = a.lse;
    p.o = static_cast<__nv_bfloat16 *>(a.o);
    p.qpos = a.qpos;
    p.status = a.status;
    const size_t smem = Smem::total + 1024;
    const cudaError_t attr_err = func_attr_once(reinterpret_cast<const void *>(attn_tc_kernel),
                                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                static_cast<int>(smem));
    if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute");
    attn_tc_kernel<<<static_cast<unsigned>(items), kThreads, smem, s>>>(tq, tk, tv, to, p);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "attention launch");
    return CS_OK;
}

}  // namespace cs
