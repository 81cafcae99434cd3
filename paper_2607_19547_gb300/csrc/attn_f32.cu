// Step 4 for fp32 storage: repair attention on the CUDA cores in fp32
// (ChronoStitch Eq. 1 restricted to the selected rows, causal in global
// sequence order).  One warp per (layer, query row, query head); keys in
// chunks of 32.
//
// Scores: the warp is four groups of eight lanes.  Group c reads keys
// j0 + 4t + c (t = 0..7) of the chunk, lane s of a group holding float4 columns
// s, s + 8, s + 16, s + 24 of the row, so every load instruction reads four whole
// 128-byte segments.  The eight partial dot products of a lane are then summed
// over its group by a halving exchange (4 + 2 + 1 shuffles), after which lane
// (c, s) holds the full score of key j0 + 4s + c.  Softmax: the chunk maximum and
// the running rescale over the warp.  Values: each lane owns float4 column `lane`
// of the output and accumulates the chunk's 32 weighted value rows (coalesced
// rows, the weight fetched from the lane that scored the key).  Every load of a
// chunk is independent of the others.
#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kWarps = 8;

__global__ void __launch_bounds__(kWarps * 32) attn_f32_kernel(AttnArgs a) {
    pdl_wait();   // inputs may come from the previous kernel of the stream
    pdl_trigger();
    const int lane = threadIdx.x & 31, grp = lane >> 3, sub = lane & 7;
    const long long wid = static_cast<long long>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
    const long long total = static_cast<long long>(a.n_layers) * a.M * a.hq;
    if (wid >= total) return;   // the same in every lane of the warp; no block barrier below
    const int h = static_cast<int>(wid % a.hq);
    const int r = static_cast<int>((wid / a.hq) % a.M);
    const int l = static_cast<int>(wid / (static_cast<long long>(a.hq) * a.M));
    const int G = a.hq / a.hkv;
    const int g = h / G;
    int qp = a.qpos[r];
    const bool bad = qp < 0 || qp >= a.T || (r > 0 && a.qpos[r - 1] >= qp);
    if (bad) {
        if (lane == 0) report_error(a.status, 5u, kSiteAttnQpos, static_cast<unsigned>(r));
        qp = min(max(qp, 0), a.T - 1);
    }
    const float4 *q4 = reinterpret_cast<const float4 *>(
        static_cast<const float *>(a.q) + (static_cast<long long>(l) * a.M + r) * a.hq * 128 + h * 128);
    const float *k = static_cast<const float *>(a.k) + static_cast<long long>(l) * a.kv_layer_stride + g * 128;
    const float *v = static_cast<const float *>(a.v) + static_cast<long long>(l) * a.kv_layer_stride + g * 128;
    float4 qf[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) qf[c] = q4[sub + 8 * c];
    const long long kstride = static_cast<long long>(a.hkv) * 128;   // floats between key rows
    const bool b2 = (sub & 4) != 0, b1 = (sub & 2) != 0, b0 = (sub & 1) != 0;
    float m = -INFINITY, den = 0.0f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int j0 = 0; j0 <= qp; j0 += 32) {
        // partial dot products of keys j0 + 4t + grp over this lane's 16 columns; a key
        // past the row's position reads the last visible key instead (in bounds, no
        // branch) and is masked after the sum
        float d[8];
#pragma unroll
        for (int t0 = 0; t0 < 8; t0 += 4) {
            float4 kv[4][4];
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                const float4 *kr = reinterpret_cast<const float4 *>(k + min(j0 + 4 * (t0 + t) + grp, qp) * kstride);
#pragma unroll
                for (int c = 0; c < 4; ++c) kv[t][c] = kr[sub + 8 * c];
            }
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                float x = 0.f, y = 0.f, z = 0.f, w = 0.f;
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    x = fmaf(qf[c].x, kv[t][c].x, x);
                    y = fmaf(qf[c].y, kv[t][c].y, y);
                    z = fmaf(qf[c].z, kv[t][c].z, z);
                    w = fmaf(qf[c].w, kv[t][c].w, w);
                }
                d[t0 + t] = (x + y) + (z + w);
            }
        }
        // halving exchange over the group's eight lanes: lane sub keeps key t = sub
        float e[4], f[2];
#pragma unroll
        for (int i = 0; i < 4; ++i)
            e[i] = (b2 ? d[i + 4] : d[i]) + __shfl_xor_sync(0xFFFFFFFFu, b2 ? d[i] : d[i + 4], 4);
#pragma unroll
        for (int i = 0; i < 2; ++i)
            f[i] = (b1 ? e[i + 2] : e[i]) + __shfl_xor_sync(0xFFFFFFFFu, b1 ? e[i] : e[i + 2], 2);
        const float dot = (b0 ? f[1] : f[0]) + __shfl_xor_sync(0xFFFFFFFFu, b0 ? f[0] : f[1], 1);
        const int j = j0 + 4 * sub + grp;   // the key whose score this lane now holds
        const float s = j <= qp ? dot * a.scale : -INFINITY;
        float mc = s;
#pragma unroll
        for (int o = 16; o >= 1; o /= 2) mc = fmaxf(mc, __shfl_xor_sync(0xFFFFFFFFu, mc, o));
        const float mn = fmaxf(m, mc);                  // finite: key j0 is always visible
        const float alpha = expf(m - mn);               // 0 on the first chunk (m = -inf)
        const float p = j <= qp ? expf(s - mn) : 0.0f;
        float ps = p;
#pragma unroll
        for (int o = 16; o >= 1; o /= 2) ps += __shfl_xor_sync(0xFFFFFFFFu, ps, o);
        den = den * alpha + ps;
        acc.x *= alpha;
        acc.y *= alpha;
        acc.z *= alpha;
        acc.w *= alpha;
        m = mn;
        const int nk = min(32, qp - j0 + 1);
#pragma unroll
        for (int i0 = 0; i0 < 32; i0 += 16) {
            float4 vv[16];   // rows past the visible keys are read clamped and not added
#pragma unroll
            for (int i = 0; i < 16; ++i)
                vv[i] = reinterpret_cast<const float4 *>(v + min(j0 + i0 + i, qp) * kstride)[lane];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                const int kk = i0 + i;   // key j0 + kk was scored by lane (kk % 4) * 8 + kk / 4
                const float pi = __shfl_sync(0xFFFFFFFFu, p, (kk & 3) * 8 + (kk >> 2));
                if (kk < nk) {
                    acc.x = fmaf(pi, vv[i].x, acc.x);
                    acc.y = fmaf(pi, vv[i].y, acc.y);
                    acc.z = fmaf(pi, vv[i].z, acc.z);
                    acc.w = fmaf(pi, vv[i].w, acc.w);
                }
            }
        }
    }
    const float inv = 1.0f / den;
    float *o = static_cast<float *>(a.o) + (static_cast<long long>(l) * a.M + r) * a.hq * 128 +
               h * 128;
    reinterpret_cast<float4 *>(o)[lane] = make_float4(acc.x * inv, acc.y * inv, acc.z * inv,
                                                      acc.w * inv);
    if (a.lse != nullptr && lane == 0)
        a.lse[(static_cast<long long>(l) * a.M + r) * a.hq + h] = m + logf(den);
}

}  // namespace

cudaError_t launch_attn_f32(const AttnArgs &a, cudaStream_t s) {
    const long long warps = static_cast<long long>(a.n_layers) * a.M * a.hq;
    if (warps == 0) return cudaSuccess;
    const long long blocks = (warps + kWarps - 1) / kWarps;
    return launch_pdl(attn_f32_kernel, dim3(static_cast<unsigned>(blocks)), dim3(kWarps * 32), 0, s, a);
}

}  // namespace cs
