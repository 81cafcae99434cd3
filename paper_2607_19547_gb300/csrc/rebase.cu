// Step 1 of the composition path: delta re-base of stored post-rotary keys
// (ChronoStitch, Eq. 3).  An HBM-bound streaming kernel: every key row of a
// moved token is read once and written once.
//
// Angles.  For token t and frequency pair i the rotation angle is
// Delta_sigma(i)(t) * theta_i with an integer Delta.  The host passes
// theta_i / (2 pi) as a 64-bit fixed-point fraction of a turn, so
// Delta * step_i (mod 2^64) is the angle reduced to one turn, exactly up to
// the 2^-64 rounding of step_i.  cos and sin of that angle are evaluated in
// double-float arithmetic (~2^-45 relative), once per distinct
// (Delta, pair) of a CTA's tokens, and kept in shared memory.
//
// Rounding.  A bf16 output is the exact rotation rounded once to bfloat16.
// The fast path evaluates x*c - y*s in fp32 with a proven error bound and
// rounds directly when no bf16 rounding midpoint lies within that bound of
// the fp32 result (Ziv's rounding test); otherwise it re-evaluates in
// double-float and rounds that.  fp32 outputs always use the double-float
// result.
#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxTokensPerCta = 32;

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

// bf16 bits of u*c - w*s, rounded once from the exact value.
__device__ __forceinline__ uint32_t rot_bf16(float u, float w, float ch, float sh,
                                             const float4 *full) {
    const float r = __fmaf_rn(u, ch, -__fmul_rn(w, sh));
    // |error of r| <= (|u| + |w|) * 2.5 * 2^-24 (product and fma roundings, plus
    // |c - ch|, |s - sh| <= 2^-25); 2^-22 leaves margin for rounding E itself.
    const float E = __fmul_rn(__fadd_rn(fabsf(u), fabsf(w)), 0x1p-22f);
    const uint32_t b = __float_as_uint(r) & 0x7FFFFFFFu;
    const uint32_t tb = b & 0x7FFF0000u;
    const float mid = __uint_as_float(tb | 0x8000u);
    const float dist = fabsf(__fsub_rn(__uint_as_float(b), mid));
    if (dist > E && __fmul_rn(E, 1024.0f) < __uint_as_float(tb) && tb < 0x7F800000u)
        return bf16_rne_bits(r);
    // double-float re-evaluation
    const float4 cs4 = *full;   // (c_hi, c_lo, s_hi, s_lo)
    const f2 p = two_prod(u, cs4.x);
    const f2 q = two_prod(w, cs4.z);
    const f2 d = two_sum(p.hi, -q.hi);
    const float tail = __fadd_rn(__fadd_rn(__fsub_rn(p.lo, q.lo), d.lo),
                                 __fsub_rn(__fmul_rn(u, cs4.y), __fmul_rn(w, cs4.w)));
    const f2 rr = two_sum(d.hi, tail);
    return bf16_round_f2(rr.hi, rr.lo);
}

// fp32 result of u*c - w*s from the double-float evaluation.
__device__ __forceinline__ float rot_f32(float u, float w, float4 cs4) {
    const f2 p = two_prod(u, cs4.x);
    const f2 q = two_prod(w, cs4.z);
    const f2 d = two_sum(p.hi, -q.hi);
    const float tail = __fadd_rn(__fadd_rn(__fsub_rn(p.lo, q.lo), d.lo),
                                 __fsub_rn(__fmul_rn(u, cs4.y), __fmul_rn(w, cs4.w)));
    return __fadd_rn(d.hi, tail);
}

// Prologue shared by both storage types: per-token deltas and the cos/sin
// table [tokens][64 pairs] in shared memory.  Returns false when no token of
// the CTA moves (nothing to rotate).
__device__ bool build_table(const RebaseArgs &a, int t0, int TB, int (*s_delta)[3],
                            float4 *tab) {
    for (int j = threadIdx.x; j < TB * 3; j += blockDim.x) {
        const int tb = j / 3, ax = j - 3 * (j / 3);
        const int t = t0 + tb;
        s_delta[tb][ax] = (t < a.T) ? a.pos_global[3 * t + ax] - a.pos_local[3 * t + ax] : 0;
    }
    __syncthreads();
    int any = 0;
    for (int j = threadIdx.x; j < TB * 3; j += blockDim.x) any |= (s_delta[j / 3][j % 3] != 0);
    if (!__syncthreads_or(any)) return false;
    // thread j: pair i = j % 64, a run of consecutive tokens; one evaluation per
    // distinct delta along the run (tokens of one chunk share their delta).
    const int groups = blockDim.x / 64;
    const int i = threadIdx.x & 63, g = threadIdx.x >> 6;
    const int per = (TB + groups - 1) / groups;
    const int axis = a.axis[i];
    const unsigned long long step = a.turn_step[i];
    int prev = 0;
    float4 val = make_float4(1.0f, 0.0f, 0.0f, 0.0f);
    bool have = false;
    for (int tb = g * per; tb < min(TB, (g + 1) * per); ++tb) {
        const int d = s_delta[tb][axis];
        if (!have || d != prev) {
            if (d == 0) {
                val = make_float4(1.0f, 0.0f, 0.0f, 0.0f);
            } else {
                f2 sn, cs;
                sincos_turns(static_cast<unsigned long long>(static_cast<long long>(d)) * step,
                             sn, cs);
                val = make_float4(cs.hi, cs.lo, sn.hi, sn.lo);
            }
            prev = d;
            have = true;
        }
        tab[tb * 64 + i] = val;
    }
    __syncthreads();
    return true;
}

// bf16: 8 threads per 128-element row, each owning 8 frequency pairs
// (16 bytes of the first half and the matching 16 bytes of the second half).
__global__ void __launch_bounds__(kThreads) rebase_bf16_kernel(RebaseArgs a, int layers_per_cta) {
    __shared__ float4 tab[kMaxTokensPerCta * 64];
    __shared__ int s_delta[kMaxTokensPerCta][3];
    const int TB = max(1, kMaxTokensPerCta / a.hkv);
    const int t0 = blockIdx.x * TB;
    const int l0 = blockIdx.y * layers_per_cta;
    const int l1 = min(a.n_layers, l0 + layers_per_cta);
    const bool moved_any = build_table(a, t0, TB, s_delta, tab);
    if (!moved_any && a.in_place) return;

    const int slot = threadIdx.x;
    if (slot >= TB * a.hkv * 8) return;
    const int tb = slot / (a.hkv * 8);
    const int h = (slot >> 3) % a.hkv;
    const int pg = slot & 7;
    const int t = t0 + tb;
    if (t >= a.T) return;
    const bool moved = (s_delta[tb][0] | s_delta[tb][1] | s_delta[tb][2]) != 0;
    if (!moved && a.in_place) return;

    const __nv_bfloat16 *src = static_cast<const __nv_bfloat16 *>(a.k_in);
    __nv_bfloat16 *dst = static_cast<__nv_bfloat16 *>(a.k_out);
    const long long row0 = (static_cast<long long>(t) * a.hkv + h) * 128 + pg * 8;
    const float4 *full = &tab[tb * 64 + pg * 8];
    float ch[8], sh[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const float4 v = full[e];
        ch[e] = v.x;
        sh[e] = v.z;
    }
    for (int l = l0; l < l1; l += 2) {
        const bool two = (l + 1 < l1);
        const long long o0 = static_cast<long long>(l) * a.layer_stride + row0;
        const long long o1 = o0 + a.layer_stride;
        uint4 x0 = __ldcs(reinterpret_cast<const uint4 *>(src + o0));
        uint4 y0 = __ldcs(reinterpret_cast<const uint4 *>(src + o0 + 64));
        uint4 x1 = make_uint4(0, 0, 0, 0), y1 = make_uint4(0, 0, 0, 0);
        if (two) {
            x1 = __ldcs(reinterpret_cast<const uint4 *>(src + o1));
            y1 = __ldcs(reinterpret_cast<const uint4 *>(src + o1 + 64));
        }
        for (int rep = 0; rep < (two ? 2 : 1); ++rep) {
            const uint4 xv = rep ? x1 : x0, yv = rep ? y1 : y0;
            const long long o = rep ? o1 : o0;
            if (!moved) {   // out-of-place copy of an unmoved token
                __stcs(reinterpret_cast<uint4 *>(dst + o), xv);
                __stcs(reinterpret_cast<uint4 *>(dst + o + 64), yv);
                continue;
            }
            const uint32_t xw[4] = {xv.x, xv.y, xv.z, xv.w};
            const uint32_t yw[4] = {yv.x, yv.y, yv.z, yv.w};
            uint32_t ow[4], pw[4];
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                const int e0 = 2 * w, e1 = 2 * w + 1;
                const float xa = bf16_lo(xw[w]), xb = bf16_hi(xw[w]);
                const float ya = bf16_lo(yw[w]), yb = bf16_hi(yw[w]);
                // first half: x c - y s ; second half: y c + x s = y c - (-x) s
                const uint32_t r0 = rot_bf16(xa, ya, ch[e0], sh[e0], full + e0);
                const uint32_t r1 = rot_bf16(xb, yb, ch[e1], sh[e1], full + e1);
                const uint32_t q0 = rot_bf16(ya, -xa, ch[e0], sh[e0], full + e0);
                const uint32_t q1 = rot_bf16(yb, -xb, ch[e1], sh[e1], full + e1);
                ow[w] = r0 | (r1 << 16);
                pw[w] = q0 | (q1 << 16);
            }
            __stcs(reinterpret_cast<uint4 *>(dst + o), make_uint4(ow[0], ow[1], ow[2], ow[3]));
            __stcs(reinterpret_cast<uint4 *>(dst + o + 64),
                   make_uint4(pw[0], pw[1], pw[2], pw[3]));
        }
    }
}

// fp32: 16 threads per 128-element row, each owning 4 frequency pairs.
__global__ void __launch_bounds__(kThreads) rebase_f32_kernel(RebaseArgs a, int layers_per_cta) {
    __shared__ float4 tab[kMaxTokensPerCta * 64];
    __shared__ int s_delta[kMaxTokensPerCta][3];
    const int TB = max(1, (kMaxTokensPerCta / 2) / a.hkv);
    const int t0 = blockIdx.x * TB;
    const int l0 = blockIdx.y * layers_per_cta;
    const int l1 = min(a.n_layers, l0 + layers_per_cta);
    const bool moved_any = build_table(a, t0, TB, s_delta, tab);
    if (!moved_any && a.in_place) return;

    const int slot = threadIdx.x;
    if (slot >= TB * a.hkv * 16) return;
    const int tb = slot / (a.hkv * 16);
    const int h = (slot >> 4) % a.hkv;
    const int pg = slot & 15;
    const int t = t0 + tb;
    if (t >= a.T) return;
    const bool moved = (s_delta[tb][0] | s_delta[tb][1] | s_delta[tb][2]) != 0;
    if (!moved && a.in_place) return;
    const float *src = static_cast<const float *>(a.k_in);
    float *dst = static_cast<float *>(a.k_out);
    const long long row0 = (static_cast<long long>(t) * a.hkv + h) * 128 + pg * 4;
    const float4 *full = &tab[tb * 64 + pg * 4];
    for (int l = l0; l < l1; ++l) {
        const long long o = static_cast<long long>(l) * a.layer_stride + row0;
        const float4 x = __ldcs(reinterpret_cast<const float4 *>(src + o));
        const float4 y = __ldcs(reinterpret_cast<const float4 *>(src + o + 64));
        if (!moved) {
            __stcs(reinterpret_cast<float4 *>(dst + o), x);
            __stcs(reinterpret_cast<float4 *>(dst + o + 64), y);
            continue;
        }
        const float xs[4] = {x.x, x.y, x.z, x.w};
        const float ys[4] = {y.x, y.y, y.z, y.w};
        float r[4], q[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float4 c = full[e];
            r[e] = rot_f32(xs[e], ys[e], c);
            q[e] = rot_f32(ys[e], -xs[e], c);
        }
        __stcs(reinterpret_cast<float4 *>(dst + o), make_float4(r[0], r[1], r[2], r[3]));
        __stcs(reinterpret_cast<float4 *>(dst + o + 64), make_float4(q[0], q[1], q[2], q[3]));
    }
}

}  // namespace

cudaError_t launch_rebase(const RebaseArgs &a, cs_dtype dt, cudaStream_t s) {
    if (a.T == 0 || a.n_layers == 0) return cudaSuccess;
    const bool bf = (dt == CS_DTYPE_BF16);
    const int TB = bf ? (a.hkv >= kMaxTokensPerCta ? 1 : kMaxTokensPerCta / a.hkv)
                      : (a.hkv >= kMaxTokensPerCta / 2 ? 1 : (kMaxTokensPerCta / 2) / a.hkv);
    const int layers_per_cta = 4;
    dim3 grid((a.T + TB - 1) / TB, (a.n_layers + layers_per_cta - 1) / layers_per_cta);
    if (bf)
        rebase_bf16_kernel<<<grid, kThreads, 0, s>>>(a, layers_per_cta);
    else
        rebase_f32_kernel<<<grid, kThreads, 0, s>>>(a, layers_per_cta);
    return cudaGetLastError();
}

}  // namespace cs
