// Step 1 of the composition path: delta re-base of stored post-rotary keys
// (ChronoStitch, Eq. 3).  An HBM-bound streaming kernel: every key row of a
// moved token is read once and written once.
//
// Angles.  For token t and frequency pair i the rotation angle is
// Delta_sigma(i)(t) * theta_i with an integer Delta.  The host passes
// theta_i / (2 pi) as a 64-bit fixed-point fraction of a turn, so
// Delta * step_i (mod 2^64) is the angle reduced to one turn, exactly up to
// the 2^-64 rounding of step_i.  cos and sin of that angle are evaluated in
// double-float arithmetic (~2^-45 relative), once per CTA for each distinct
// token delta, and kept in shared memory.
//
// Rounding.  A bf16 output is the exact rotation rounded once to bfloat16.
// The fast path evaluates x*c - y*s in fp32 with a proven error bound and
// rounds directly when no bf16 rounding midpoint lies within that bound of
// the fp32 result (Ziv's rounding test); otherwise it re-evaluates in
// double-float and rounds that.  fp32 outputs always use the double-float
// result.
#include <algorithm>

#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxTokensPerCta = 32;   // fp32 kernel
constexpr int kMaxTokensBf16 = 16;     // bf16 kernel: token block of 16 / n_kv_heads
constexpr int kMaxBlocks = 512;        // 8-element blocks of one token row (32 kv heads)

// 1/n! split exactly into fp32 hi + lo (hi = fp32(1/n!), lo = fp32(1/n! - hi)).
__device__ __forceinline__ f2 cf(float hi, float lo) { return {hi, lo}; }

// cos and sin of (u / 2^64) turns, as double-float values.
__device__ void sincos_turns(unsigned long long u, f2 &sn, f2 &cs) {
    // nearest quarter turn q and the residual v in [-2^61, 2^61) units of 2^-64 turns
    const unsigned long long qq = (u + (1ull << 61)) >> 62;
    const long long v = static_cast<long long>(u - (qq << 62));
    const unsigned q = static_cast<unsigned>(qq) & 3u;
    const float vh = __ll2float_rn(v);
    const float vl = __ll2float_rn(v - static_cast<long long>(vh));
    const f2 vv = fast_two_sum(vh, vl);
    // x = v * 2 pi / 2^64 radians, |x| <= pi/4
    const f2 two_pi_scaled = {0x1.921fb6p-62f, -0x1.777a5cp-87f};
    const f2 x = df_mul(vv, two_pi_scaled);
    const f2 z = df_mul(x, x);
    const float zf = z.hi;

    // sin x = x * sum_k (-1)^k z^k / (2k+1)!  ; terms k >= 5 are below 2^-28 and stay in fp32
    float ts = __fmaf_rn(__fmaf_rn(-0x1.ae7f3ep-41f, zf, 0x1.612462p-33f), zf, -0x1.ae6456p-26f);
    f2 p = {ts, 0.0f};
    p = df_add(df_mul(p, z), cf(0x1.71de3ap-19f, 0x1.55b1ccp-45f));     //  1/9!
    p = df_add(df_mul(p, z), cf(-0x1.a01a02p-13f, 0x1.7f97fap-39f));    // -1/7!
    p = df_add(df_mul(p, z), cf(0x1.111112p-7f, -0x1.dddddep-32f));     //  1/5!
    p = df_add(df_mul(p, z), cf(-0x1.555556p-3f, 0x1.555556p-28f));     // -1/3!
    p = df_add(df_mul(p, z), cf(1.0f, 0.0f));
    const f2 s = df_mul(x, p);

    // cos x = sum_k (-1)^k z^k / (2k)!  ; terms k >= 5 in fp32
    float tc = __fmaf_rn(__fmaf_rn(__fmaf_rn(0x1.ae7f3ep-45f, zf, -0x1.93974ap-37f), zf,
                                   0x1.1eed8ep-29f), zf, -0x1.27e4fcp-22f);
    f2 r = {tc, 0.0f};
    r = df_add(df_mul(r, z), cf(0x1.a01a02p-16f, -0x1.7f97fap-42f));    //  1/8!
    r = df_add(df_mul(r, z), cf(-0x1.6c16c2p-10f, 0x1.27d27ep-35f));    // -1/6!
    r = df_add(df_mul(r, z), cf(0x1.555556p-5f, -0x1.555556p-30f));     //  1/4!
    r = df_add(df_mul(r, z), cf(-0.5f, 0.0f));                          // -1/2!
    r = df_add(df_mul(r, z), cf(1.0f, 0.0f));
    const f2 c = r;

    const f2 ns = {-s.hi, -s.lo}, nc = {-c.hi, -c.lo};
    switch (q) {
        case 0: sn = s;  cs = c;  break;
        case 1: sn = c;  cs = ns; break;
        case 2: sn = ns; cs = nc; break;
        default: sn = nc; cs = s; break;
    }
}

// bf16 bits of u*c - w*s from the double-float evaluation (c = c_hi + c_lo,
// s = s_hi + s_lo), rounded once: the error-free products and sum carry the
// value to about 2^-44 relative, far inside any rounding decision left to it.
// When the leading sum already overflows fp32 (|p - q| >= 2^128 - 2^103), the
// exact value lies beyond the bf16 overflow threshold 2^128 - 2^119 as well,
// so the result is that infinity (the error terms would turn into NaN).
__device__ __forceinline__ uint32_t rot_bf16_df(float u, float w, float4 cs4) {
    const f2 p = two_prod(u, cs4.x);
    const f2 q = two_prod(w, cs4.z);
    const f2 d = two_sum(p.hi, -q.hi);
    if (isinf(d.hi)) return __float_as_uint(d.hi) >> 16;
    const float tail = __fadd_rn(__fadd_rn(__fsub_rn(p.lo, q.lo), d.lo),
                                 __fsub_rn(__fmul_rn(u, cs4.y), __fmul_rn(w, cs4.w)));
    const f2 rr = two_sum(d.hi, tail);
    return bf16_round_f2(rr.hi, rr.lo);
}

// Slices whose bf16 rounding was uncertain wait in a per-warp queue in shared
// memory (their raw input words and where they came from) and are redone by the
// whole warp together, one output pair per lane, so the rare slow path never runs
// on one lane while the other 31 wait.
constexpr int kQueue = 48;   // entries per warp

__shared__ uint4 q_xy[kThreads / 32][2 * kQueue];   // first- and second-half words
__shared__ uint32_t q_meta[kThreads / 32][kQueue];  // (slice index << 5) | owning lane

// Rotates the n queued slices of this warp entirely in double-float, rounds each
// output once and stores it.  Called by exactly the lanes of `part` (the lanes
// that rotate), each passing its own output offset `obase` and table row `trow`.
__device__ __forceinline__ void redo_queue(int n, unsigned part, long long obase,
                                        long long lstep, int trow, const float4 *tab,
                                        __nv_bfloat16 *dst) {
    __syncwarp(part);   // entries written by other lanes
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int rank = __popc(part & ((1u << lane) - 1u));
    const int nl = __popc(part);
    const int items = n * 8;   // 8 frequency pairs per slice
    uint16_t *d16 = reinterpret_cast<uint16_t *>(dst);
    for (int base = 0; base < items; base += nl) {   // the same trip count on every lane
        const int it = base + rank;
        const bool valid = it < items;
        const int ent = valid ? it >> 3 : 0, p = it & 7;
        const uint32_t mt = q_meta[warp][ent];
        const int olane = static_cast<int>(mt & 31u);
        const long long ob = __shfl_sync(part, obase, olane);
        const int orow = __shfl_sync(part, trow, olane);
        if (valid) {
            const uint32_t *w = reinterpret_cast<const uint32_t *>(&q_xy[warp][2 * ent]);
            const uint32_t xw = w[p >> 1], yw = w[4 + (p >> 1)];
            const float x = (p & 1) ? bf16_hi(xw) : bf16_lo(xw);
            const float y = (p & 1) ? bf16_hi(yw) : bf16_lo(yw);
            const float4 cs4 = tab[orow + p];
            const long long o = ob + static_cast<long long>(mt >> 5) * lstep + p;
            d16[o] = static_cast<uint16_t>(rot_bf16_df(x, y, cs4));
            d16[o + 64] = static_cast<uint16_t>(rot_bf16_df(y, -x, cs4));
        }
    }
    __syncwarp(part);   // the queue is reused; later reads of these rows see the stores
}

// Two fp32 values rounded to nearest-even bf16 and packed (lo in bits 0-15).
__device__ __forceinline__ uint32_t pack_bf16x2_rn(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// Per-thread staging of the next layers' input words in shared memory with 16-byte
// asynchronous copies (cp.async, bypassing L1): kStages layers of every thread's two
// words are in flight without holding registers.  Each thread copies and later reads
// only its own slots, so the copies need no block barrier: a wait on the thread's own
// copy groups makes them visible to it.  Slot (stage s, half h) of thread x sits at
// word (s * 2 + h) * kThreads + x, so a warp's reads and copies touch consecutive
// 16-byte words.  Six stages (48 KB) with the cos/sin table beside them leave room
// for three CTAs per SM; measured on the 3B shapes against four stages at four CTAs
// per SM, and against three, five and eight stages, six was the fastest at every size.
constexpr int kStages = 6;
constexpr size_t kStageBytes = static_cast<size_t>(kStages) * 2 * kThreads * 16;

__device__ __forceinline__ uint4 *stage_slot(uint4 *buf, int s, int h) {
    return buf + (s * 2 + h) * kThreads + threadIdx.x;
}
__device__ __forceinline__ void cp_async16(uint4 *smem, const void *gmem) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem)), "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}
// Waits until at most kStages - 1 of this thread's copy groups are still in flight
// (groups complete in order, so every older group is complete).
__device__ __forceinline__ void cp_async_wait_stage() {
    asm volatile("cp.async.wait_group %0;" ::"n"(kStages - 1) : "memory");
}

// fp32 result of u*c - w*s from the double-float evaluation (an overflowing
// leading sum is returned as the infinity it rounds to, as above).
__device__ __forceinline__ float rot_f32(float u, float w, float4 cs4) {
    const f2 p = two_prod(u, cs4.x);
    const f2 q = two_prod(w, cs4.z);
    const f2 d = two_sum(p.hi, -q.hi);
    if (isinf(d.hi)) return d.hi;
    const float tail = __fadd_rn(__fadd_rn(__fsub_rn(p.lo, q.lo), d.lo),
                                 __fsub_rn(__fmul_rn(u, cs4.y), __fmul_rn(w, cs4.w)));
    return __fadd_rn(d.hi, tail);
}

// Prologue shared by both storage types: per-token deltas and the cos/sin
// table [tokens][64 pairs] in shared memory.  Tokens of one chunk share their
// delta, so when every token of the block has the same delta the 64 entries
// are evaluated once and copied.  Returns false when no token of the block
// moves (nothing to rotate).
__device__ bool build_table(const RebaseArgs &a, int t0, int TB, int (*s_delta)[3],
                            float4 *tab) {
    for (int j = threadIdx.x; j < TB * 3; j += blockDim.x) {
        const int tb = j / 3, ax = j - 3 * (j / 3);
        const int t = t0 + tb;
        s_delta[tb][ax] = (t < a.T) ? a.pos_global[3 * t + ax] - a.pos_local[3 * t + ax] : 0;
    }
    __syncthreads();
    int any = 0, same = 1;
    for (int j = threadIdx.x; j < TB * 3; j += blockDim.x) {
        any |= (s_delta[j / 3][j % 3] != 0);
        same &= (s_delta[j / 3][j % 3] == s_delta[0][j % 3]);
    }
    any = __syncthreads_or(any);
    same = __syncthreads_and(same);
    if (!any) return false;
    const int ntok = same ? 1 : TB;
    for (int j = threadIdx.x; j < ntok * 64; j += blockDim.x) {
        const int tb = j >> 6, i = j & 63;
        const int d = s_delta[tb][a.axis[i]];
        float4 val = make_float4(1.0f, 0.0f, 0.0f, 0.0f);
        if (d != 0) {
            f2 sn, cs;
            sincos_turns(static_cast<unsigned long long>(static_cast<long long>(d)) * a.turn_step[i],
                         sn, cs);
            val = make_float4(cs.hi, cs.lo, sn.hi, sn.lo);
        }
        if (same) {
            for (int q = 0; q < TB; ++q) tab[q * 64 + i] = val;
        } else {
            tab[tb * 64 + i] = val;
        }
    }
    __syncthreads();
    return true;
}

// Rotates one thread's slice: 8 frequency pairs, i.e. 16-byte words xv (first
// half: elements i) and yv (second half: elements i + 64).  Returns false if
// the bf16 rounding of any output is uncertain.
//
// Each output r ~ u c - w s is evaluated in fp32 with
//   |r - exact| <= 2.5 * 2^-24 * (|x| + |y|) + 2^-149
// (c_hi and s_hi lie within 2^-25 of cos and sin; one rounding of the product,
// one of the fma; the last term covers subnormal results).  With
//   E = fl(4 * 2^-24 * fl(|x| + |y|) + 2^-147),
// lo = fl(r - E) and hi = fl(r + E) bracket the exact value: E exceeds the error
// bound by 1.5 * 2^-24 (|x| + |y|) + 2^-148, more than the rounding error of either
// sum (at most 2^-24 (|r| + E), or 2^-150 for subnormal sums).  Rounding to nearest
// (ties to even) is monotone, so when lo and hi round to the same bf16 value the
// exact value rounds to it too, and so does r (lo <= r <= hi).  The test is
// therefore: round lo and hi of two adjacent outputs with one packed conversion
// each and compare the two words.  A non-finite input or an overflowing sum makes
// lo and hi differ (an infinity meets a NaN or the other infinity), except a NaN
// input, whose NaN output is accepted as it is.
__device__ __forceinline__ bool rotate_slice(const uint4 &xv, const uint4 &yv, const float (&c)[8],
                                             const float (&sn)[8], uint32_t (&ow)[4],
                                             uint32_t (&pw)[4]) {
    const uint32_t xw[4] = {xv.x, xv.y, xv.z, xv.w};
    const uint32_t yw[4] = {yv.x, yv.y, yv.z, yv.w};
    const float2 kE = make_float2(0x1p-22f, 0x1p-22f);       // 4 * 2^-24
    const float2 kT = make_float2(0x1p-147f, 0x1p-147f);
    const float2 kM = make_float2(-1.0f, -1.0f);
    uint32_t diff = 0;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const int e0 = 2 * w, e1 = 2 * w + 1;
        const float x0 = bf16_lo(xw[w]), x1 = bf16_hi(xw[w]);
        const float y0 = bf16_lo(yw[w]), y1 = bf16_hi(yw[w]);
        // two frequency pairs at once in packed fp32 (the same roundings as one pair at a
        // time: one product, then one fused multiply-add)
        const float2 X = make_float2(x0, x1), Y = make_float2(y0, y1);
        const float2 C = make_float2(c[e0], c[e1]), S = make_float2(sn[e0], sn[e1]);
        const float2 ys = __fmul2_rn(Y, S), xs = __fmul2_rn(X, S);
        const float2 r1 = __ffma2_rn(X, C, make_float2(-ys.x, -ys.y));   // x c - y s
        const float2 r2 = __ffma2_rn(Y, C, xs);                          // y c + x s
        const float2 u = make_float2(__fadd_rn(fabsf(x0), fabsf(y0)), __fadd_rn(fabsf(x1), fabsf(y1)));
        const float2 E = __ffma2_rn(u, kE, kT);
        const float2 lo1 = __ffma2_rn(E, kM, r1), hi1 = __fadd2_rn(r1, E);
        const float2 lo2 = __ffma2_rn(E, kM, r2), hi2 = __fadd2_rn(r2, E);
        diff |= pack_bf16x2_rn(lo1.x, lo1.y) ^ pack_bf16x2_rn(hi1.x, hi1.y);
        diff |= pack_bf16x2_rn(lo2.x, lo2.y) ^ pack_bf16x2_rn(hi2.x, hi2.y);
        ow[w] = pack_bf16x2_rn(r1.x, r1.y);
        pw[w] = pack_bf16x2_rn(r2.x, r2.y);
    }
    return diff == 0;
}

// Eq. 5 block term of the canonical fp32 order: ((q0+q1)+(q2+q3))+((q4+q5)+(q6+q7)),
// q = (fresh - cached)^2 rounded at every step, for one 16-byte word of each side.
__device__ __forceinline__ float score_block8(uint4 fv, uint4 cv) {
    const uint32_t fw[4] = {fv.x, fv.y, fv.z, fv.w};
    const uint32_t cw[4] = {cv.x, cv.y, cv.z, cv.w};
    float q[8];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const float d0 = __fsub_rn(bf16_lo(fw[w]), bf16_lo(cw[w]));
        const float d1 = __fsub_rn(bf16_hi(fw[w]), bf16_hi(cw[w]));
        q[2 * w] = __fmul_rn(d0, d0);
        q[2 * w + 1] = __fmul_rn(d1, d1);
    }
    return __fadd_rn(__fadd_rn(__fadd_rn(q[0], q[1]), __fadd_rn(q[2], q[3])),
                     __fadd_rn(__fadd_rn(q[4], q[5]), __fadd_rn(q[6], q[7])));
}

// Eq. 5's fixed halving order over one token's block sums s[0..B) in shared memory,
// by one warp: the sums are padded with +0 to a power of two P >= 32 (x + 0 = x for the
// non-negative block sums, so padding past the canonical power of two changes
// nothing), lane l holds s[l + 32 j], strides >= 32 are folded in-lane and strides 16
// .. 1 by an xor butterfly (s[b] + s[b ^ m] = s[b] + s[b + m] for b < m).  Returns the
// score in every lane.
__device__ __forceinline__ float reduce_blocks_warp(const float *blk, int B) {
    constexpr int kMaxJ = kMaxBlocks / 32;
    const int lane = threadIdx.x & 31;
    int P = 32;
    while (P < B) P *= 2;
    float v[kMaxJ];
#pragma unroll
    for (int j = 0; j < kMaxJ; ++j) v[j] = (32 * j < P && lane + 32 * j < B) ? blk[lane + 32 * j] : 0.0f;
#pragma unroll
    for (int m = kMaxJ / 2; m >= 1; m /= 2) {
        if (32 * m < P) {
#pragma unroll
            for (int j = 0; j < m; ++j) v[j] = __fadd_rn(v[j], v[j + m]);
        }
    }
    float r = v[0];
#pragma unroll
    for (int m = 16; m >= 1; m /= 2) r = __fadd_rn(r, __shfl_xor_sync(0xFFFFFFFFu, r, m));
    return r;
}

// The streaming part of the bf16 kernel for one thread's slices (see the kernel
// below).  `part` holds the lanes of this warp that rotate (moved tokens with
// layers to walk); they all walk the same number of layers.  The first kStages
// layers' words were requested by the kernel (stage_first); every iteration waits
// for its stage, uses it, and requests the layer kStages further on into it.
__device__ __forceinline__ void stream_slices(const __nv_bfloat16 *src, __nv_bfloat16 *dst,
                                              long long obase, long long lstep, int count,
                                              bool moved, unsigned part, int trow,
                                              const float4 *tab, uint4 *stage) {
    int s = 0;   // stage holding layer i
    if (!moved) {   // out-of-place copy of an unmoved token
        for (int i = 0; i < count; ++i) {
            cp_async_wait_stage();
            const uint4 xv = *stage_slot(stage, s, 0), yv = *stage_slot(stage, s, 1);
            const long long o = obase + i * lstep;
            __stcs(reinterpret_cast<uint4 *>(dst + o), xv);
            __stcs(reinterpret_cast<uint4 *>(dst + o + 64), yv);
            if (i + kStages < count) {
                cp_async16(stage_slot(stage, s, 0), src + o + kStages * lstep);
                cp_async16(stage_slot(stage, s, 1), src + o + kStages * lstep + 64);
            }
            cp_async_commit();
            s = s + 1 == kStages ? 0 : s + 1;
        }
        return;
    }
    const float4 *full = &tab[trow];
    float c[8], sn[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        c[e] = full[e].x;
        sn[e] = full[e].z;
    }
    int queued = 0;   // the same on every lane of `part`
#pragma unroll 1
    for (int i = 0; i < count; ++i) {
        if (queued > kQueue - 32) {   // make room for one failing slice per lane
            redo_queue(queued, part, obase, lstep, trow, tab, dst);
            queued = 0;
        }
        cp_async_wait_stage();
        const uint4 xv = *stage_slot(stage, s, 0), yv = *stage_slot(stage, s, 1);
        uint32_t ow[4], pw[4];
        const bool ok = rotate_slice(xv, yv, c, sn, ow, pw);
        const long long o = obase + i * lstep;
        if (ok) {
            __stcs(reinterpret_cast<uint4 *>(dst + o), make_uint4(ow[0], ow[1], ow[2], ow[3]));
            __stcs(reinterpret_cast<uint4 *>(dst + o + 64), make_uint4(pw[0], pw[1], pw[2], pw[3]));
        }
        const unsigned fails = __ballot_sync(part, !ok);
        if (fails) {   // rare: queue the uncertain slices (not stored) for the warp to redo
            if (!ok) {
                const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
                const int e = queued + __popc(fails & ((1u << lane) - 1u));
                q_xy[warp][2 * e] = xv;
                q_xy[warp][2 * e + 1] = yv;
                q_meta[warp][e] = (static_cast<uint32_t>(i) << 5) | static_cast<uint32_t>(lane);
            }
            queued += __popc(fails);
        }
        // the stage's words have been used (stored or queued): request the layer kStages
        // further on into it
        if (i + kStages < count) {
            cp_async16(stage_slot(stage, s, 0), src + o + kStages * lstep);
            cp_async16(stage_slot(stage, s, 1), src + o + kStages * lstep + 64);
        }
        cp_async_commit();
        s = s + 1 == kStages ? 0 : s + 1;
    }
    if (queued) redo_queue(queued, part, obase, lstep, trow, tab, dst);
}

// bf16: 8 threads per 128-element row, each owning 8 frequency pairs (16 bytes
// of the first half and the matching 16 bytes of the second half).  A CTA
// takes a block of TB tokens (TB * n_kv_heads * 8 threads per layer "slot")
// and walks every layer of its range, n_slots layers at a time, so the cos/sin
// table of its tokens is built once and reused across layers.
//   - each thread reads its own token's delta and issues its first load before
//     the table is built, so DRAM latency overlaps the sincos evaluation;
//   - the next layer's slice is loaded before the current one is rotated;
//   - a slice with an uncertain rounding is not stored; its input words go to
//     the warp's redo queue and the whole warp redoes the queued slices in
//     double-float when the queue fills and after the streaming loop;
//   - with the fused score, the slot that re-based layer score_layer reads its
//     candidate rows back (its own stores) with the matching fresh rows and
//     reduces each token's 16 * n_kv_heads block sums in the canonical halving
//     order: token rows are adjacent lanes of one warp (8 lanes per head), so
//     strides of 16 and more blocks are lane offsets of 8 and 16, the stride of
//     8 blocks stays inside a thread (its two halves), and 4, 2, 1 are lane
//     offsets again.
// HKV > 0: the kv head count is that compile-time constant (the token block is
// then 16 / HKV tokens, 128 threads per layer slot, two slots, and the index
// arithmetic below is shifts); HKV == 0: any head count, TB as passed.  Two slots
// (each thread walks half of the CTA's layers) measured faster than four at every
// size: half as many CTA prologues, and longer per-thread streams.
// Dynamic shared memory: the kStages staging buffers, then the table (TB * 64 entries).
template <int HKV>
__global__ void __launch_bounds__(kThreads, 3) rebase_bf16_kernel(RebaseArgs a, int TB_arg, int l_per_cta) {
    pdl_wait();   // inputs may come from the previous kernel of the stream
    pdl_trigger();
    const int hkv = HKV > 0 ? HKV : a.hkv;
    const int TB = HKV > 0 ? 16 / HKV : TB_arg;
    extern __shared__ uint4 stage[];
    float4 *tab = reinterpret_cast<float4 *>(stage + kStages * 2 * kThreads);
    __shared__ int s_delta[kMaxTokensBf16][3];
    const int t0 = blockIdx.x * TB;
    const int l0 = blockIdx.y * l_per_cta;
    const int l1 = min(a.n_layers, l0 + l_per_cta);
    const int slot_threads = TB * hkv * 8;
    const int n_slots = kThreads / slot_threads;
    const int slot = threadIdx.x / slot_threads;
    const int loc = threadIdx.x - slot * slot_threads;
    const int tb = loc / (hkv * 8);
    const int h = (loc >> 3) % hkv;
    const int pg = loc & 7;
    const int t = t0 + tb;
    const int lfirst = l0 + slot;
    bool mine = (slot < n_slots) && (t < a.T) && (lfirst < l1);
    bool moved = false;
    if (mine) {
        moved = ((a.pos_global[3 * t] - a.pos_local[3 * t]) |
                 (a.pos_global[3 * t + 1] - a.pos_local[3 * t + 1]) |
                 (a.pos_global[3 * t + 2] - a.pos_local[3 * t + 2])) != 0;
        if (!moved && a.in_place) mine = false;
    }
    const int count = mine ? (l1 - lfirst + n_slots - 1) / n_slots : 0;
    const __nv_bfloat16 *src = static_cast<const __nv_bfloat16 *>(a.k_in);
    __nv_bfloat16 *dst = static_cast<__nv_bfloat16 *>(a.k_out);
    const long long row0 = (static_cast<long long>(t) * hkv + h) * 128 + pg * 8;
    const long long lstep = static_cast<long long>(n_slots) * a.layer_stride;
    const long long obase = static_cast<long long>(lfirst) * a.layer_stride + row0;
    // the first layers' words go out before the table is built (empty groups past count)
    for (int st = 0; st < kStages; ++st) {
        if (st < count) {
            cp_async16(stage_slot(stage, st, 0), src + obase + st * lstep);
            cp_async16(stage_slot(stage, st, 1), src + obase + st * lstep + 64);
        }
        cp_async_commit();
    }
    const bool moved_any = build_table(a, t0, TB, s_delta, tab);
    const bool scoring = a.score_out != nullptr && slot < n_slots && t < a.T && t >= a.cand0 &&
                         t < a.cand0 + a.n_cand && a.score_layer >= l0 && a.score_layer < l1 &&
                         (a.score_layer - l0) % n_slots == slot;
    // build_table ended with a block barrier: every lane takes part in this ballot
    const unsigned part = __ballot_sync(0xFFFFFFFFu, count > 0 && moved && moved_any);
    if (count > 0)
        stream_slices(src, dst, obase, lstep, count, moved, part, tb * 64 + pg * 8, tab, stage);
    if (HKV == 0) {
        // any head count: a token's row may span several warps, so its block sums meet in
        // shared memory and one warp per token reduces them in the canonical order
        const bool cta_scores = a.score_out != nullptr && a.score_layer >= l0 &&
                                a.score_layer < l1 && t0 < a.cand0 + a.n_cand &&
                                t0 + TB > a.cand0;
        if (!cta_scores) return;   // the same in every thread of the CTA
        __shared__ float s_blk[kMaxBlocks];
        const int B = 16 * hkv;    // blocks of one token row (TB * B <= kMaxBlocks)
        if (scoring) {
            const long long o = static_cast<long long>(a.score_layer) * a.layer_stride + row0;
            const uint4 cx = *reinterpret_cast<const uint4 *>(dst + o);
            const uint4 cy = *reinterpret_cast<const uint4 *>(dst + o + 64);
            const __nv_bfloat16 *fr = static_cast<const __nv_bfloat16 *>(a.fresh) +
                                      static_cast<long long>(t - a.cand0) * a.fresh_stride + h * 128 + pg * 8;
            s_blk[tb * B + h * 16 + pg] = score_block8(__ldg(reinterpret_cast<const uint4 *>(fr)), cx);
            s_blk[tb * B + h * 16 + 8 + pg] =
                score_block8(__ldg(reinterpret_cast<const uint4 *>(fr + 64)), cy);
        }
        __syncthreads();
        for (int tk = threadIdx.x >> 5; tk < TB; tk += kThreads / 32) {
            const int tt = t0 + tk;
            if (tt < a.T && tt >= a.cand0 && tt < a.cand0 + a.n_cand) {   // uniform over the warp
                const float v = reduce_blocks_warp(&s_blk[tk * B], B);
                if ((threadIdx.x & 31) == 0) a.score_out[tt - a.cand0] = v;
            }
        }
        return;
    }
    if (a.score_out == nullptr || __ballot_sync(0xFFFFFFFFu, scoring) == 0) return;
    float s1 = 0.0f, s2 = 0.0f;
    if (scoring) {
        const long long o = static_cast<long long>(a.score_layer) * a.layer_stride + row0;
        const uint4 cx = *reinterpret_cast<const uint4 *>(dst + o);
        const uint4 cy = *reinterpret_cast<const uint4 *>(dst + o + 64);
        const __nv_bfloat16 *fr = static_cast<const __nv_bfloat16 *>(a.fresh) +
                                  static_cast<long long>(t - a.cand0) * a.fresh_stride + h * 128 + pg * 8;
        s1 = score_block8(__ldg(reinterpret_cast<const uint4 *>(fr)), cx);
        s2 = score_block8(__ldg(reinterpret_cast<const uint4 *>(fr + 64)), cy);
    }
    for (int m = 8 * hkv; m >= 16; m /= 2) {   // block strides >= 16: heads h and h + m/16
        s1 = __fadd_rn(s1, __shfl_down_sync(0xFFFFFFFFu, s1, m / 2));
        s2 = __fadd_rn(s2, __shfl_down_sync(0xFFFFFFFFu, s2, m / 2));
    }
    s1 = __fadd_rn(s1, s2);   // stride 8: the two halves of a head
#pragma unroll
    for (int m = 4; m >= 1; m /= 2) s1 = __fadd_rn(s1, __shfl_down_sync(0xFFFFFFFFu, s1, m));
    if (scoring && h == 0 && pg == 0) a.score_out[t - a.cand0] = s1;
}

// fp32: 16 threads per 128-element row, each owning 4 frequency pairs.  With the
// fused score, the CTA whose layer range holds score_layer scores its candidate
// tokens from the re-based values it holds in registers: each thread's four squared
// differences of a half form one half of an 8-element block (((q0+q1)+(q2+q3)) from
// the even thread, ((q4+q5)+(q6+q7)) from the odd one, joined by one shuffle), the
// block sums meet in shared memory and one warp per token reduces them in the
// canonical order.
__global__ void __launch_bounds__(kThreads) rebase_f32_kernel(RebaseArgs a, int layers_per_cta) {
    pdl_wait();   // inputs may come from the previous kernel of the stream
    pdl_trigger();
    __shared__ float4 tab[kMaxTokensPerCta * 64];
    __shared__ int s_delta[kMaxTokensPerCta][3];
    __shared__ float s_blk[kMaxBlocks];
    const int TB = max(1, (kMaxTokensPerCta / 2) / a.hkv);
    const int t0 = blockIdx.x * TB;
    const int l0 = blockIdx.y * layers_per_cta;
    const int l1 = min(a.n_layers, l0 + layers_per_cta);
    const bool moved_any = build_table(a, t0, TB, s_delta, tab);
    const bool cta_scores = a.score_out != nullptr && a.score_layer >= l0 && a.score_layer < l1 &&
                            t0 < a.cand0 + a.n_cand && t0 + TB > a.cand0;
    if (!moved_any && a.in_place && !cta_scores) return;   // the same in every thread

    const int slot = threadIdx.x;
    const int tb = slot / (a.hkv * 16);
    const int h = (slot >> 4) % a.hkv;
    const int pg = slot & 15;
    const int t = t0 + tb;
    const bool active = slot < TB * a.hkv * 16 && t < a.T;
    const bool moved = active && (s_delta[tb][0] | s_delta[tb][1] | s_delta[tb][2]) != 0;
    const bool writes = active && (moved || !a.in_place);
    const bool scoring = cta_scores && active && t >= a.cand0 && t < a.cand0 + a.n_cand;
    const float *src = static_cast<const float *>(a.k_in);
    float *dst = static_cast<float *>(a.k_out);
    const long long row0 = (static_cast<long long>(t) * a.hkv + h) * 128 + pg * 4;
    const float4 *full = &tab[tb * 64 + pg * 4];
    float px = 0.0f, py = 0.0f;   // this thread's halves of its two score blocks
    for (int l = l0; l < l1; ++l) {
        const bool sc = scoring && l == a.score_layer;
        if (!writes && !sc) continue;
        const long long o = static_cast<long long>(l) * a.layer_stride + row0;
        const float4 x = __ldcs(reinterpret_cast<const float4 *>(src + o));
        const float4 y = __ldcs(reinterpret_cast<const float4 *>(src + o + 64));
        float r[4] = {x.x, x.y, x.z, x.w};
        float q[4] = {y.x, y.y, y.z, y.w};
        if (moved) {
            const float xs[4] = {x.x, x.y, x.z, x.w};
            const float ys[4] = {y.x, y.y, y.z, y.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float4 c = full[e];
                r[e] = rot_f32(xs[e], ys[e], c);
                q[e] = rot_f32(ys[e], -xs[e], c);
            }
        }
        if (writes) {
            __stcs(reinterpret_cast<float4 *>(dst + o), make_float4(r[0], r[1], r[2], r[3]));
            __stcs(reinterpret_cast<float4 *>(dst + o + 64), make_float4(q[0], q[1], q[2], q[3]));
        }
        if (sc) {
            const float *fr = static_cast<const float *>(a.fresh) +
                              static_cast<long long>(t - a.cand0) * a.fresh_stride + h * 128 + pg * 4;
            const float4 fx = __ldg(reinterpret_cast<const float4 *>(fr));
            const float4 fy = __ldg(reinterpret_cast<const float4 *>(fr + 64));
            const float f1[4] = {fx.x, fx.y, fx.z, fx.w}, f2[4] = {fy.x, fy.y, fy.z, fy.w};
            float d1[4], d2[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float u = __fsub_rn(f1[e], r[e]), v = __fsub_rn(f2[e], q[e]);
                d1[e] = __fmul_rn(u, u);
                d2[e] = __fmul_rn(v, v);
            }
            px = __fadd_rn(__fadd_rn(d1[0], d1[1]), __fadd_rn(d1[2], d1[3]));
            py = __fadd_rn(__fadd_rn(d2[0], d2[1]), __fadd_rn(d2[2], d2[3]));
        }
    }
    if (!cta_scores) return;   // the same in every thread
    // block sum = (even thread's half) + (odd thread's half); x + y = y + x exactly
    const float ox = __shfl_xor_sync(0xFFFFFFFFu, px, 1);
    const float oy = __shfl_xor_sync(0xFFFFFFFFu, py, 1);
    const int B = 16 * a.hkv;     // blocks of one token row (TB * B <= kMaxBlocks)
    if (scoring && (pg & 1) == 0) {
        s_blk[tb * B + h * 16 + (pg >> 1)] = __fadd_rn(px, ox);
        s_blk[tb * B + h * 16 + 8 + (pg >> 1)] = __fadd_rn(py, oy);
    }
    __syncthreads();
    for (int tk = threadIdx.x >> 5; tk < TB; tk += kThreads / 32) {
        const int tt = t0 + tk;
        if (tt < a.T && tt >= a.cand0 && tt < a.cand0 + a.n_cand) {   // uniform over the warp
            const float v = reduce_blocks_warp(&s_blk[tk * B], B);
            if ((threadIdx.x & 31) == 0) a.score_out[tt - a.cand0] = v;
        }
    }
}

}  // namespace

bool rebase_fuses_score(const RebaseArgs &a, cs_dtype dt) {
    // every head count the kernels take (bf16 up to 32, fp32 up to 16 kv heads)
    return (dt == CS_DTYPE_BF16 && a.hkv <= 32) || (dt == CS_DTYPE_F32 && a.hkv <= 16);
}

cudaError_t launch_rebase(const RebaseArgs &a, cs_dtype dt, cudaStream_t s) {
    if (a.T == 0 || a.n_layers == 0) return cudaSuccess;
    if (dt == CS_DTYPE_BF16) {
        // token block: 128 threads per layer slot where possible (2 slots per CTA)
        const int TB = a.hkv >= kMaxTokensBf16 ? 1 : kMaxTokensBf16 / a.hkv;
        const int blocks = (a.T + TB - 1) / TB;
        const int slots = kThreads / (TB * a.hkv * 8);
        // split layers across CTAs only when there are too few token blocks to fill
        // the GPU (every extra CTA repeats the cos/sin prologue)
        int groups = 1;
        const int sms = sm_count();
        const int target = (sms > 0 ? sms : 152) * 2;
        if (blocks < target) groups = std::min((target + blocks - 1) / blocks,
                                               (a.n_layers + slots - 1) / slots);
        const int l_per_cta = (a.n_layers + groups - 1) / groups;
        dim3 grid(blocks, (a.n_layers + l_per_cta - 1) / l_per_cta);
        const size_t smem = kStageBytes + static_cast<size_t>(TB) * 64 * sizeof(float4);
        auto *kern = a.hkv == 1 ? rebase_bf16_kernel<1> : a.hkv == 2 ? rebase_bf16_kernel<2>
                   : a.hkv == 4 ? rebase_bf16_kernel<4> : rebase_bf16_kernel<0>;
        // the limit covers the largest table, so one setting serves every head count
        constexpr size_t kSmemMax = kStageBytes + kMaxTokensBf16 * 64 * sizeof(float4);
        const cudaError_t attr_err = func_attr_once(reinterpret_cast<const void *>(kern),
                                                    cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                    static_cast<int>(kSmemMax));
        if (attr_err != cudaSuccess) return attr_err;
        return launch_pdl(kern, grid, dim3(kThreads), smem, s, a, TB, l_per_cta);
    } else {
        const int TB = a.hkv >= kMaxTokensPerCta / 2 ? 1 : (kMaxTokensPerCta / 2) / a.hkv;
        const int layers_per_cta = 4;
        dim3 grid((a.T + TB - 1) / TB, (a.n_layers + layers_per_cta - 1) / layers_per_cta);
        return launch_pdl(rebase_f32_kernel, grid, dim3(kThreads), 0, s, a, layers_per_cta);
    }
    return cudaGetLastError();
}

}  // namespace cs
