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
// CTA = 6 warps:
//   warp 0      TMA producer: Q once, then K and V tiles through an
//               NS-stage shared-memory ring (128-byte swizzle).
//   warp 1      owns tensor memory; lane 0 issues tcgen05.mma:
//               S_j = Q K_j^T  (A, B from shared memory, fp32 into TMEM,
//               double-buffered), O += P_j V_j (A = P from TMEM, B = V from
//               shared memory, MN-major).
//   warps 2-5   softmax: thread = one TMEM lane = one query row.  Reads S_j,
//               masks, updates the running max (rescaling O in TMEM only
//               when the max grows by more than 2^8), writes P_j = exp2(...)
//               as bf16 over the first 64 columns of S_j's TMEM buffer,
//               and finally normalises O and stores it.
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

constexpr int kThreads = 192;
constexpr int kBlockN = 128;           // keys per KV tile
constexpr int kStages = 2;             // K/V shared-memory ring depth
constexpr uint32_t kTileBytes = 128 * 128 * 2;      // one K or V tile (two 16 KB halves)
constexpr uint32_t kHalfBytes = 128 * 64 * 2;
constexpr uint32_t kTmemCols = 512;    // S0 [0,128) S1 [128,256) O [256,384)
constexpr uint32_t kColO = 256;
constexpr uint64_t kWaitLimitNs = 1000000000ull;    // 1 s

struct Smem {
    // byte offsets from the 1024-aligned base
    static constexpr uint32_t q = 0;
    static constexpr uint32_t k = q + kTileBytes;
    static constexpr uint32_t v = k + kStages * kTileBytes;
    static constexpr uint32_t bars = v + kStages * kTileBytes;
    static constexpr uint32_t total = bars + 256;
};

struct Bars {
    uint64_t q_full;
    uint64_t k_full[kStages], k_empty[kStages];
    uint64_t v_full[kStages], v_empty[kStages];
    uint64_t s_full[2], p_full[2];
    uint64_t o_done;     // one completion per P*V block
    uint64_t o_final;    // single use: every P*V of the tile is done
    uint64_t mma_done;   // single use: every tensor-core operation of the CTA retired
    uint32_t tmem_base;
    int abort;
};
static_assert(sizeof(Bars) <= 256, "barrier area");

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

// Tile coordinates of work item `item`, heaviest query tiles first (selected
// rows are ascending, so later query tiles see more keys).
__device__ __forceinline__ void decode_item(const TcParams &p, int item, int &l, int &g, int &qt) {
    const int per = p.n_layers * p.hkv;
    qt = p.n_qtiles - 1 - item / per;
    const int rem = item % per;
    l = rem / p.hkv;
    g = rem % p.hkv;
}

__device__ __forceinline__ int clamp_pos(int x, int T) { return min(max(x, 0), T - 1); }

__global__ void __launch_bounds__(kThreads, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
               const __grid_constant__ CUtensorMap tm_v, const TcParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *base = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    Bars *bars = reinterpret_cast<Bars *>(base + Smem::bars);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    int l, g, qt;
    decode_item(p, blockIdx.x, l, g, qt);
    const int r0 = qt * p.tok;
    const int r_last = min(p.M, r0 + p.tok) - 1;
    const int qmin = clamp_pos(p.qpos[r0], p.T);
    const int kmax = clamp_pos(p.qpos[r_last], p.T);
    const int nb = kmax / kBlockN + 1;
    const int mask_from = qmin / kBlockN;
    const uint32_t q_bytes = static_cast<uint32_t>(p.tok * p.G) * 256u;   // both 64-column halves

    if (threadIdx.x == 0) {
        mbar_init(&bars->q_full, 1);
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&bars->k_full[s], 1);
            mbar_init(&bars->k_empty[s], 1);
            mbar_init(&bars->v_full[s], 1);
            mbar_init(&bars->v_empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars->s_full[b], 1);
            mbar_init(&bars->p_full[b], 128);
        }
        mbar_init(&bars->o_done, 1);
        mbar_init(&bars->o_final, 1);
        mbar_init(&bars->mma_done, 1);
        bars->abort = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&bars->tmem_base, kTmemCols);
        tmem_relinquish();
    }
    // rows of the Q tile that TMA does not write (G not dividing 128) must be finite
    {
        const uint32_t used = static_cast<uint32_t>(p.tok * p.G) * 128u;   // bytes per half
        for (uint32_t off = used + threadIdx.x * 16u; off < kHalfBytes; off += kThreads * 16u) {
            *reinterpret_cast<uint4 *>(base + Smem::q + off) = make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4 *>(base + Smem::q + kHalfBytes + off) = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async_smem();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int *abort = &bars->abort;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&tm_q);
            tma_prefetch_desc(&tm_k);
            tma_prefetch_desc(&tm_v);
            mbar_arrive_expect_tx(&bars->q_full, q_bytes);
            tma_load_4d(base + Smem::q, &tm_q, &bars->q_full, 0, g * p.G, r0, l);
            tma_load_4d(base + Smem::q + kHalfBytes, &tm_q, &bars->q_full, 64, g * p.G, r0, l);
            int nk = 0, nv = 0;   // K and V tiles issued
            for (int j = 0; j < nb; ++j) {
                const int s = j % kStages;
                const uint32_t ph = (j / kStages) & 1;
                if (!mbar_wait_bounded(&bars->k_empty[s], ph ^ 1, abort, p.status,
                                       kSiteAttnProducer, kWaitLimitNs)) break;
                uint8_t *kd = base + Smem::k + s * kTileBytes;
                mbar_arrive_expect_tx(&bars->k_full[s], kTileBytes);
                tma_load_4d(kd, &tm_k, &bars->k_full[s], 0, g, j * kBlockN, l);
                tma_load_4d(kd + kHalfBytes, &tm_k, &bars->k_full[s], 64, g, j * kBlockN, l);
                ++nk;
                if (!mbar_wait_bounded(&bars->v_empty[s], ph ^ 1, abort, p.status,
                                       kSiteAttnProducer, kWaitLimitNs)) break;
                uint8_t *vd = base + Smem::v + s * kTileBytes;
                mbar_arrive_expect_tx(&bars->v_full[s], kTileBytes);
                tma_load_4d(vd, &tm_v, &bars->v_full[s], 0, g, j * kBlockN, l);
                tma_load_4d(vd + kHalfBytes, &tm_v, &bars->v_full[s], 64, g, j * kBlockN, l);
                ++nv;
            }
            if (*abort) {
                // drain: every issued copy lands before the CTA's shared memory is released.
                // Phases of one barrier complete in order, so waiting for the last
                // copy issued on each barrier covers the earlier ones.
                volatile int never = 0;
                mbar_wait_bounded(&bars->q_full, 0, &never, nullptr, 0, kWaitLimitNs);
                for (int s = 0; s < kStages; ++s) {
                    for (int which = 0; which < 2; ++which) {
                        const int cnt = which ? nv : nk;
                        if (cnt <= s) continue;
                        const int jl = s + ((cnt - 1 - s) / kStages) * kStages;
                        uint64_t *bar = which ? &bars->v_full[s] : &bars->k_full[s];
                        mbar_wait_bounded(bar, (jl / kStages) & 1, &never, nullptr, 0,
                                          kWaitLimitNs);
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            const uint32_t idesc_qk = idesc_bf16(128, 128, 0, 0);
            const uint32_t idesc_pv = idesc_bf16(128, 128, 0, 1);
            const uint32_t q_addr = smem_u32(base + Smem::q);
            bool ok = mbar_wait_bounded(&bars->q_full, 0, abort, p.status, kSiteAttnMma,
                                        kWaitLimitNs);
            auto issue_qk = [&](int j) -> bool {
                const int s = j % kStages;
                if (!mbar_wait_bounded(&bars->k_full[s], (j / kStages) & 1, abort, p.status,
                                       kSiteAttnMma, kWaitLimitNs)) return false;
                tc_fence_after();
                const uint32_t k_addr = smem_u32(base + Smem::k + s * kTileBytes);
                const uint32_t d = tmem + static_cast<uint32_t>((j & 1) * 128);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint32_t off = (kk >> 2) * kHalfBytes + (kk & 3) * 32;
                    tc_mma_ss(d, smem_desc(q_addr + off, 16, 1024, 2),
                              smem_desc(k_addr + off, 16, 1024, 2), idesc_qk, kk > 0);
                }
                tc_commit(&bars->s_full[j & 1]);
                tc_commit(&bars->k_empty[s]);
                return true;
            };
            if (ok) ok = issue_qk(0);
            for (int j = 0; ok && j < nb; ++j) {
                if (j + 1 < nb) {
                    // S_{j+1} overwrites the buffer that held P_{j-1}: PV_{j-1} must be done
                    if (j >= 1 && !mbar_wait_bounded(&bars->o_done, (j - 1) & 1, abort, p.status,
                                                     kSiteAttnMma, kWaitLimitNs)) { ok = false; break; }
                    if (!issue_qk(j + 1)) { ok = false; break; }
                }
                const int s = j % kStages;
                if (!mbar_wait_bounded(&bars->p_full[j & 1], (j >> 1) & 1, abort, p.status,
                                       kSiteAttnMma, kWaitLimitNs)) { ok = false; break; }
                if (!mbar_wait_bounded(&bars->v_full[s], (j / kStages) & 1, abort, p.status,
                                       kSiteAttnMma, kWaitLimitNs)) { ok = false; break; }
                tc_fence_after();
                const uint32_t v_addr = smem_u32(base + Smem::v + s * kTileBytes);
                const uint32_t a_tm = tmem + static_cast<uint32_t>((j & 1) * 128);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    // A: 16 keys of P = 8 packed columns; B: 16 rows (keys) of V, MN-major
                    tc_mma_ts(tmem + kColO, a_tm + kk * 8,
                              smem_desc(v_addr + kk * 2048, kHalfBytes, 1024, 2), idesc_pv,
                              (j > 0 || kk > 0) ? 1u : 0u);
                }
                tc_commit(&bars->o_done);
                tc_commit(&bars->v_empty[s]);
                if (j == nb - 1) tc_commit(&bars->o_final);
            }
            // completes once every tcgen05 operation issued above has retired
            tc_commit(&bars->mma_done);
        }
    } else {
        // ------------------------------------------------------------ softmax
        const int qw = warp & 3;
        const int m = 32 * qw + lane;                 // TMEM lane = MMA row
        const int t = m / p.G, hh = m - t * p.G;
        const int r = r0 + t;
        const bool valid = (m < p.tok * p.G) && (r <= r_last);
        int qp = kmax;
        if (valid) {
            const int raw = p.qpos[r];
            if (raw < 0 || raw >= p.T || (r > 0 && p.qpos[r - 1] >= raw))
                report_error(p.status, 5u, kSiteAttnQpos, static_cast<unsigned>(r));
            qp = clamp_pos(raw, p.T);
        }
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * qw) << 16);
        float m_run = -INFINITY, l_run = 0.0f;
        bool ok = true;
        for (int j = 0; j < nb; ++j) {
            const int b = j & 1;
            const bool w_ok = mbar_wait_bounded(&bars->s_full[b], (j >> 1) & 1, abort, p.status,
                                                kSiteAttnSoftmax, kWaitLimitNs);
            if (!__all_sync(0xFFFFFFFFu, w_ok)) { ok = false; *abort = 1; break; }
            tc_fence_after();
            float s[128];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t rr[32];
                tmem_ld32(lane_base + b * 128 + c * 32, rr);
#pragma unroll
                for (int e = 0; e < 32; ++e) s[c * 32 + e] = __uint_as_float(rr[e]);
            }
            if (j >= mask_from) {
                const int lim = qp - j * kBlockN;
#pragma unroll
                for (int c = 0; c < 128; ++c)
                    if (c > lim) s[c] = -INFINITY;
            }
            float mx = s[0];
#pragma unroll
            for (int c = 1; c < 128; ++c) mx = fmaxf(mx, s[c]);
            const float mx2 = mx * p.scale_log2;
            const bool grow = (m_run == -INFINITY) || (mx2 > m_run + 8.0f);
            float alpha = 1.0f;
            if (grow) {
                alpha = exp2f(m_run - mx2);   // 0 on the first block
                l_run *= alpha;
                m_run = mx2;
            }
            // P_j = exp2(s * scale * log2(e) - m_run), packed bf16 over columns [0, 64)
            float psum = 0.0f;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t pk[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const float p0 = __uint_as_float(ex2_approx(__fmaf_rn(s[c * 32 + 2 * e], p.scale_log2, -m_run)));
                    const float p1 = __uint_as_float(ex2_approx(__fmaf_rn(s[c * 32 + 2 * e + 1], p.scale_log2, -m_run)));
                    psum += p0 + p1;
                    pk[e] = pack_bf16x2(p0, p1);
                }
                tmem_st16(lane_base + b * 128 + c * 16, pk);
            }
            l_run += psum;
            // rescale O when any row of this warp raised its max (O holds PV_0..PV_{j-1})
            if (j > 0 && __any_sync(0xFFFFFFFFu, grow)) {
                const bool o_ok = mbar_wait_bounded(&bars->o_done, (j - 1) & 1, abort, p.status,
                                                    kSiteAttnSoftmax, kWaitLimitNs);
                if (!__all_sync(0xFFFFFFFFu, o_ok)) { ok = false; *abort = 1; break; }
                tc_fence_after();
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    uint32_t rr[32];
                    tmem_ld32(lane_base + kColO + c * 32, rr);
#pragma unroll
                    for (int e = 0; e < 32; ++e)
                        rr[e] = __float_as_uint(__uint_as_float(rr[e]) * alpha);
                    tmem_st32(lane_base + kColO + c * 32, rr);
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
        if (ok) {
            tc_fence_after();
            const float inv = 1.0f / l_run;
            __nv_bfloat16 *orow = p.o + ((static_cast<long long>(l) * p.M + r) * p.hq + g * p.G + hh) * 128;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t rr[32];
                tmem_ld32(lane_base + kColO + c * 32, rr);
                if (valid) {
                    uint32_t pk[16];
#pragma unroll
                    for (int e = 0; e < 16; ++e)
                        pk[e] = pack_bf16x2(__uint_as_float(rr[2 * e]) * inv,
                                            __uint_as_float(rr[2 * e + 1]) * inv);
                    uint4 *dst = reinterpret_cast<uint4 *>(orow + c * 32);
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        dst[e] = make_uint4(pk[4 * e], pk[4 * e + 1], pk[4 * e + 2], pk[4 * e + 3]);
                }
            }
            if (valid && p.lse != nullptr)
                p.lse[(static_cast<long long>(l) * p.M + r) * p.hq + g * p.G + hh] =
                    (m_run + __log2f(l_run)) * 0.69314718055994531f;
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
    CUtensorMap tq, tk, tv;
    const cuuint64_t qdims[4] = {128, static_cast<cuuint64_t>(a.hq), static_cast<cuuint64_t>(a.M),
                                 static_cast<cuuint64_t>(a.n_layers)};
    const cuuint64_t qstr[3] = {256ull, 256ull * a.hq, 256ull * a.hq * a.M};
    const cuuint32_t qbox[4] = {64, static_cast<cuuint32_t>(G), static_cast<cuuint32_t>(tok), 1};
    const cuuint64_t kdims[4] = {128, static_cast<cuuint64_t>(a.hkv), static_cast<cuuint64_t>(a.T),
                                 static_cast<cuuint64_t>(a.n_layers)};
    const cuuint64_t kstr[3] = {256ull, 256ull * a.hkv, 2ull * static_cast<cuuint64_t>(a.kv_layer_stride)};
    const cuuint32_t kbox[4] = {64, 1, 128, 1};
    if (!make_map(enc, &tq, a.q, qdims, qstr, qbox) || !make_map(enc, &tk, a.k, kdims, kstr, kbox) ||
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
    static std::once_flag attr_once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(attr_once, [&] {
        attr_err = cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        static_cast<int>(smem));
    });
    if (attr_err != cudaSuccess) return cuda_fail(attr_err, "cudaFuncSetAttribute");
    attn_tc_kernel<<<static_cast<unsigned>(items), kThreads, smem, s>>>(tq, tk, tv, p);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "attention launch");
    return CS_OK;
}

}  // namespace cs
