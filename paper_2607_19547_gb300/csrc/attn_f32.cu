// Step 4 for fp32 storage: repair attention on the CUDA cores in fp32
// (ChronoStitch Eq. 1 restricted to the selected rows, causal in global
// sequence order).  One warp per (layer, query row, query head); each lane
// owns 4 of the 128 dimensions.  Online softmax over keys 0..qpos[r].
#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {
namespace {

constexpr int kWarps = 8;

__global__ void __launch_bounds__(kWarps * 32) attn_f32_kernel(AttnArgs a) {
    pdl_wait();   // inputs may come from the previous kernel of the stream
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const long long wid = static_cast<long long>(blockIdx.x) * kWarps + (threadIdx.x >> 5);
    const long long total = static_cast<long long>(a.n_layers) * a.M * a.hq;
    if (wid >= total) return;
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
    const float *q = static_cast<const float *>(a.q) + (static_cast<long long>(l) * a.M + r) *
                                                          a.hq * 128 + h * 128;
    const float *k = static_cast<const float *>(a.k) + static_cast<long long>(l) * a.kv_layer_stride;
    const float *v = static_cast<const float *>(a.v) + static_cast<long long>(l) * a.kv_layer_stride;
    const float4 qv = reinterpret_cast<const float4 *>(q)[lane];
    float m = -INFINITY, den = 0.0f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int j = 0; j <= qp; ++j) {
        const long long off = (static_cast<long long>(j) * a.hkv + g) * 128;
        const float4 kv = reinterpret_cast<const float4 *>(k + off)[lane];
        float part = qv.x * kv.x + qv.y * kv.y + qv.z * kv.z + qv.w * kv.w;
#pragma unroll
        for (int o = 16; o >= 1; o /= 2) part += __shfl_xor_sync(0xFFFFFFFFu, part, o);
        const float s = part * a.scale;
        const float4 vv = reinterpret_cast<const float4 *>(v + off)[lane];
        if (s > m) {
            const float alpha = expf(m - s);   // 0 on the first key (m = -inf)
            den = den * alpha + 1.0f;
            acc.x = acc.x * alpha + vv.x;
            acc.y = acc.y * alpha + vv.y;
            acc.z = acc.z * alpha + vv.z;
            acc.w = acc.w * alpha + vv.w;
            m = s;
        } else {
            const float p = expf(s - m);
            den += p;
            acc.x += p * vv.x;
            acc.y += p * vv.y;
            acc.z += p * vv.z;
            acc.w += p * vv.w;
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
