// C ABI entry points of libchronostitch: argument validation on the host,
// kernel launches, and the per-device status word that kernels write when
// they detect a data error or a bounded wait gives up.
#include <cuda.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {

// Per-device status area (static storage of this module, one copy per device).
__device__ __align__(16) unsigned int g_status[kStatusWords];

namespace {

thread_local char t_detail[512] = "no error";

constexpr int kMaxDevices = 64;
std::mutex g_mu;
unsigned int *g_status_addr[kMaxDevices] = {};
CUcontext g_status_ctx[kMaxDevices] = {};
std::mutex g_take_mu;   // one take at a time: the take slot (words 2-3) is shared

using CtxGetCurrentFn = CUresult (*)(CUcontext *);

// The driver's cuCtxGetCurrent, through the runtime's entry-point query (no link
// against the driver library); nullptr if unavailable.
CtxGetCurrentFn ctx_get_current_fn() {
    static CtxGetCurrentFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &ptr, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<CtxGetCurrentFn>(ptr);
    });
    return fn;
}

CUcontext current_ctx() {
    CUcontext c = nullptr;
    CtxGetCurrentFn fn = ctx_get_current_fn();
    if (fn == nullptr || fn(&c) != CUDA_SUCCESS) return nullptr;
    return c;
}

cudaStream_t as_stream(void *s) { return static_cast<cudaStream_t>(s); }

// theta_i / (2 pi) in units of 2^-64 turns, rounded to nearest, from the fp64
// value of theta_i = theta^(-2i/D).  theta_i = m * 2^e exactly (m < 2^53); the
// product with round(2^66 / (2 pi)) is formed in 128-bit integer arithmetic.
unsigned long long turn_step(double theta_i) {
    int e;
    const double fr = std::frexp(theta_i, &e);                    // theta_i = fr * 2^e, fr in [0.5,1)
    const unsigned long long m = static_cast<unsigned long long>(std::ldexp(fr, 53));  // exact
    e -= 53;                                                       // theta_i = m * 2^e
    const unsigned __int128 inv2pi_66 = 0xa2f9836e4e44152aull;     // round(2^66 / (2 pi))
    const unsigned __int128 prod = static_cast<unsigned __int128>(m) * inv2pi_66;
    // step = prod * 2^(e - 2); theta_i <= 1 gives e <= -53, a right shift of >= 55
    const int sh = 2 - e;
    if (sh >= 128) return 0;
    const unsigned __int128 half = static_cast<unsigned __int128>(1) << (sh - 1);
    return static_cast<unsigned long long>((prod + half) >> sh);
}

}  // namespace

cs_status fail(cs_status s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    std::vsnprintf(t_detail, sizeof(t_detail), fmt, ap);
    va_end(ap);
    return s;
}

cs_status cuda_fail(cudaError_t e, const char *what) {
    return fail(CS_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

unsigned int *status_word() {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        cuda_fail(e, "cudaGetDevice");
        return nullptr;
    }
    if (dev < 0 || dev >= kMaxDevices) {
        fail(CS_ERR_UNSUPPORTED, "device ordinal %d beyond %d", dev, kMaxDevices);
        return nullptr;
    }
    // the address belongs to the context the module was loaded in: after a device reset
    // (a new primary context) it is looked up again
    const CUcontext ctx = current_ctx();
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_status_addr[dev] == nullptr || ctx == nullptr || g_status_ctx[dev] != ctx) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_status);
        if (e != cudaSuccess) {
            cuda_fail(e, "cudaGetSymbolAddress(status word)");
            return nullptr;
        }
        g_status_addr[dev] = static_cast<unsigned int *>(p);
        g_status_ctx[dev] = current_ctx();   // the look-up may have created the context
    }
    return g_status_addr[dev];
}

cudaError_t func_attr_once(const void *fn, cudaFuncAttribute attr, int value) {
    struct Entry {
        const void *fn;
        int dev;
        int attr;
        int value;
        cudaError_t err;
    };
    static std::mutex mu;
    static Entry done[64];
    static int n_done = 0;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < n_done; ++i)
        if (done[i].fn == fn && done[i].dev == dev && done[i].attr == static_cast<int>(attr) &&
            done[i].value == value)
            return done[i].err;
    e = cudaFuncSetAttribute(fn, attr, value);
    if (n_done < 64) done[n_done++] = Entry{fn, dev, static_cast<int>(attr), value, e};
    return e;
}

int sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    return n;
}

}  // namespace cs

using namespace cs;

extern "C" {

int cs_abi_version(void) { return 1; }

const char *cs_status_string(cs_status s) {
    switch (s) {
        case CS_OK: return "ok";
        case CS_ERR_INVALID_ARG: return "invalid argument";
        case CS_ERR_UNSUPPORTED: return "unsupported configuration";
        case CS_ERR_CUDA: return "CUDA error";
        case CS_ERR_TIMEOUT: return "device wait timed out";
        case CS_ERR_DEVICE_ARG: return "device data check failed";
    }
    return "unknown status";
}

const char *cs_last_error_detail(void) { return t_detail; }

namespace {

// [a, a + an) and [b, b + bn) (bytes) share an address
bool overlaps(const void *a, long long an, const void *b, long long bn) {
    const char *x = static_cast<const char *>(a);
    const char *y = static_cast<const char *>(b);
    return x < y + bn && y < x + an;
}

// The layer-`score_layer` score requested together with a re-base.
struct ScoreRequest {
    int score_layer, cand0, n_cand;
    const void *fresh;
    long long fresh_stride;
    float *score_out;
};

cs_status rebase_impl(const void *k_in, void *k_out, cs_dtype dtype, int n_layers,
                      int64_t layer_stride, int T, int n_kv_heads, int head_dim,
                      const int32_t *pos_local, const int32_t *pos_global, const cs_rope_cfg *rope,
                      const ScoreRequest *sc, void *stream) {
    if (dtype != CS_DTYPE_F32 && dtype != CS_DTYPE_BF16) return fail(CS_ERR_INVALID_ARG, "dtype");
    if (n_layers < 0 || T < 0 || n_kv_heads <= 0 || head_dim <= 0)
        return fail(CS_ERR_INVALID_ARG, "negative size or non-positive head count/dim");
    if (head_dim != 128) return fail(CS_ERR_UNSUPPORTED, "head_dim %d (only 128)", head_dim);
    const int max_heads = dtype == CS_DTYPE_BF16 ? 32 : 16;
    if (n_kv_heads > max_heads)
        return fail(CS_ERR_UNSUPPORTED, "n_kv_heads %d > %d", n_kv_heads, max_heads);
    if (rope == nullptr) return fail(CS_ERR_INVALID_ARG, "rope config is NULL");
    if (!(std::isfinite(rope->theta) && rope->theta > 1.0))
        return fail(CS_ERR_INVALID_ARG, "rope theta must be finite and > 1");
    long long ssum = 0;
    for (int a = 0; a < 3; ++a) {
        if (rope->sections[a] < 0) return fail(CS_ERR_INVALID_ARG, "negative mrope section");
        ssum += rope->sections[a];
    }
    if (ssum != head_dim / 2)
        return fail(CS_ERR_INVALID_ARG, "mrope sections sum to %lld, need %d", ssum, head_dim / 2);
    const long long row = static_cast<long long>(n_kv_heads) * head_dim;
    if (layer_stride < static_cast<long long>(T) * row)
        return fail(CS_ERR_INVALID_ARG, "layer_stride %lld < T*n_kv_heads*head_dim",
                    static_cast<long long>(layer_stride));
    const long long esz = dtype == CS_DTYPE_BF16 ? 2 : 4;
    const bool scoring = sc != nullptr && sc->n_cand > 0;
    if (sc != nullptr) {
        if (sc->n_cand < 0 || sc->cand0 < 0 || static_cast<long long>(sc->cand0) + sc->n_cand > T)
            return fail(CS_ERR_INVALID_ARG, "candidates [cand0, cand0 + n_cand) must lie in [0, T)");
        if (scoring && (sc->score_layer < 0 || sc->score_layer >= n_layers))
            return fail(CS_ERR_INVALID_ARG, "score_layer %d outside [0, %d)", sc->score_layer, n_layers);
        if (row > 2048) return fail(CS_ERR_UNSUPPORTED, "row of %lld elements > 2048", row);
        if (sc->fresh_stride < row)
            return fail(CS_ERR_INVALID_ARG, "fresh row stride shorter than n_kv_heads*head_dim");
        if (scoring && (sc->fresh == nullptr || sc->score_out == nullptr))
            return fail(CS_ERR_INVALID_ARG, "NULL fresh keys or score output");
        if (scoring && (!aligned16(sc->fresh) || (sc->fresh_stride * esz) % 16))
            return fail(CS_ERR_INVALID_ARG, "fresh rows must start 16-byte aligned");
        if (scoring && n_layers > 0 && T > 0) {
            const long long out_bytes = 4ll * sc->n_cand;
            const long long keys_bytes = ((n_layers - 1) * layer_stride + T * row) * esz;
            const long long fresh_bytes = ((sc->n_cand - 1) * sc->fresh_stride + row) * esz;
            if (overlaps(sc->score_out, out_bytes, k_in, keys_bytes) ||
                overlaps(sc->score_out, out_bytes, k_out, keys_bytes) ||
                overlaps(sc->score_out, out_bytes, sc->fresh, fresh_bytes))
                return fail(CS_ERR_INVALID_ARG, "score_out overlaps the keys");
            if (overlaps(sc->fresh, fresh_bytes, k_out, keys_bytes))
                return fail(CS_ERR_INVALID_ARG, "k_fresh overlaps the re-based keys");
        }
    }
    if (n_layers == 0 || T == 0) return CS_OK;
    if (k_in == nullptr || k_out == nullptr || pos_local == nullptr || pos_global == nullptr)
        return fail(CS_ERR_INVALID_ARG, "NULL tensor pointer");
    if (!aligned16(k_in) || !aligned16(k_out) || (layer_stride * esz) % 16)
        return fail(CS_ERR_INVALID_ARG, "keys must be 16-byte aligned (pointers and layer stride)");
    const long long key_span = ((n_layers - 1) * layer_stride + T * row) * esz;
    if (k_in != k_out && overlaps(k_in, key_span, k_out, key_span))
        return fail(CS_ERR_INVALID_ARG, "k_in and k_out overlap without being equal");
    {
        // every CTA reads its tokens' coordinates while others write keys (and scores)
        const long long pos_bytes = 12ll * T;
        if (overlaps(pos_local, pos_bytes, k_out, key_span) ||
            overlaps(pos_global, pos_bytes, k_out, key_span))
            return fail(CS_ERR_INVALID_ARG, "coordinates overlap the re-based keys");
        if (scoring && (overlaps(pos_local, pos_bytes, sc->score_out, 4ll * sc->n_cand) ||
                        overlaps(pos_global, pos_bytes, sc->score_out, 4ll * sc->n_cand)))
            return fail(CS_ERR_INVALID_ARG, "coordinates overlap score_out");
    }
    RebaseArgs args;
    std::memset(&args, 0, sizeof(args));
    args.k_in = k_in;
    args.k_out = k_out;
    args.n_layers = n_layers;
    args.layer_stride = layer_stride;
    args.T = T;
    args.hkv = n_kv_heads;
    args.pos_local = pos_local;
    args.pos_global = pos_global;
    args.in_place = (k_in == k_out);
    int i = 0;
    for (int a = 0; a < 3; ++a)
        for (int c = 0; c < rope->sections[a]; ++c, ++i) args.axis[i] = static_cast<unsigned char>(a);
    for (i = 0; i < head_dim / 2; ++i)
        args.turn_step[i] = turn_step(std::pow(rope->theta, -(2.0 * i) / head_dim));
    if (scoring) {
        args.fresh = sc->fresh;
        args.fresh_stride = sc->fresh_stride;
        args.score_out = sc->score_out;
        args.score_layer = sc->score_layer;
        args.cand0 = sc->cand0;
        args.n_cand = sc->n_cand;
        if (!rebase_fuses_score(args, dtype)) args.score_out = nullptr;   // scored below
    }
    cudaError_t e = launch_rebase(args, dtype, as_stream(stream));
    if (e != cudaSuccess) return cuda_fail(e, "rebase launch");
    if (scoring && args.score_out == nullptr) {
        const char *cached = static_cast<const char *>(k_out) +
                             (static_cast<long long>(sc->score_layer) * layer_stride +
                              static_cast<long long>(sc->cand0) * row) * esz;
        e = launch_score(sc->fresh, cached, dtype, sc->n_cand, static_cast<int>(row), sc->fresh_stride,
                         row, sc->score_out, as_stream(stream));
        if (e != cudaSuccess) return cuda_fail(e, "score launch");
    }
    return CS_OK;
}

}  // namespace

cs_status cs_rebase_keys(const void *k_in, void *k_out, cs_dtype dtype, int n_layers,
                         int64_t layer_stride, int T, int n_kv_heads, int head_dim,
                         const int32_t *pos_local, const int32_t *pos_global,
                         const cs_rope_cfg *rope, void *stream) {
    return rebase_impl(k_in, k_out, dtype, n_layers, layer_stride, T, n_kv_heads, head_dim, pos_local,
                       pos_global, rope, nullptr, stream);
}

cs_status cs_rebase_and_score(const void *k_in, void *k_out, cs_dtype dtype, int n_layers,
                              int64_t layer_stride, int T, int n_kv_heads, int head_dim,
                              const int32_t *pos_local, const int32_t *pos_global,
                              const cs_rope_cfg *rope, int score_layer, int cand0, int n_cand,
                              const void *k_fresh, int64_t fresh_row_stride, float *score_out,
                              void *stream) {
    const ScoreRequest sc{score_layer, cand0, n_cand, k_fresh, fresh_row_stride, score_out};
    return rebase_impl(k_in, k_out, dtype, n_layers, layer_stride, T, n_kv_heads, head_dim, pos_local,
                       pos_global, rope, &sc, stream);
}

cs_status cs_score_deviation(const void *k_fresh, const void *k_cached, cs_dtype dtype, int n,
                             int n_kv_heads, int head_dim, int64_t fresh_row_stride,
                             int64_t cached_row_stride, float *score_out, void *stream) {
    if (dtype != CS_DTYPE_F32 && dtype != CS_DTYPE_BF16) return fail(CS_ERR_INVALID_ARG, "dtype");
    if (n < 0 || n_kv_heads <= 0 || head_dim <= 0)
        return fail(CS_ERR_INVALID_ARG, "negative size or non-positive head count/dim");
    if (head_dim != 128) return fail(CS_ERR_UNSUPPORTED, "head_dim %d (only 128)", head_dim);
    const long long E = static_cast<long long>(n_kv_heads) * head_dim;
    if (E > 2048) return fail(CS_ERR_UNSUPPORTED, "row of %lld elements > 2048", E);
    if (fresh_row_stride < E || cached_row_stride < E)
        return fail(CS_ERR_INVALID_ARG, "row stride shorter than n_kv_heads*head_dim");
    if (n == 0) return CS_OK;
    if (k_fresh == nullptr || k_cached == nullptr || score_out == nullptr)
        return fail(CS_ERR_INVALID_ARG, "NULL pointer");
    const long long esz = dtype == CS_DTYPE_BF16 ? 2 : 4;
    if (!aligned16(k_fresh) || !aligned16(k_cached) || (fresh_row_stride * esz) % 16 ||
        (cached_row_stride * esz) % 16)
        return fail(CS_ERR_INVALID_ARG, "rows must start 16-byte aligned");
    if (overlaps(score_out, 4ll * n, k_fresh, ((n - 1) * fresh_row_stride + E) * esz) ||
        overlaps(score_out, 4ll * n, k_cached, ((n - 1) * cached_row_stride + E) * esz))
        return fail(CS_ERR_INVALID_ARG, "score_out overlaps the keys");
    const cudaError_t e = launch_score(k_fresh, k_cached, dtype, n, static_cast<int>(E),
                                       fresh_row_stride, cached_row_stride, score_out,
                                       as_stream(stream));
    if (e != cudaSuccess) return cuda_fail(e, "score launch");
    return CS_OK;
}

cs_status cs_select_topk(const float *score, int n, int k, int32_t idx_base, int32_t *out_idx,
                         void *stream) {
    if (n < 0 || k < 0 || k > n) return fail(CS_ERR_INVALID_ARG, "need 0 <= k <= n (n=%d k=%d)", n, k);
    if (idx_base < 0 || static_cast<long long>(idx_base) + n > 0x7FFFFFFFll)
        return fail(CS_ERR_INVALID_ARG, "idx_base + n must stay within int32");
    if (k == 0) return CS_OK;
    if (score == nullptr || out_idx == nullptr) return fail(CS_ERR_INVALID_ARG, "NULL pointer");
    {
        // the indices are written while scores may still be read (large n re-reads them)
        const char *sc = reinterpret_cast<const char *>(score);
        const char *oc = reinterpret_cast<const char *>(out_idx);
        if (oc < sc + 4ll * n && sc < oc + 4ll * k)
            return fail(CS_ERR_INVALID_ARG, "out_idx overlaps score");
    }
    const cudaError_t e = launch_select(score, n, k, idx_base, out_idx, as_stream(stream));
    if (e != cudaSuccess) return cuda_fail(e, "select launch");
    return CS_OK;
}

cs_status cs_scatter_rows(void *cache, const void *rows, cs_dtype dtype, int n_layers, int T,
                          int64_t cache_layer_stride, int n_rows, int64_t rows_layer_stride,
                          int row_elems, const int32_t *idx, void *stream) {
    if (dtype != CS_DTYPE_F32 && dtype != CS_DTYPE_BF16) return fail(CS_ERR_INVALID_ARG, "dtype");
    if (n_layers < 0 || T < 0 || n_rows < 0 || row_elems <= 0)
        return fail(CS_ERR_INVALID_ARG, "negative size or non-positive row_elems");
    const long long esz = dtype == CS_DTYPE_BF16 ? 2 : 4;
    if ((row_elems * esz) % 16)
        return fail(CS_ERR_UNSUPPORTED, "row bytes %lld not a multiple of 16", row_elems * esz);
    if (cache_layer_stride < static_cast<long long>(T) * row_elems)
        return fail(CS_ERR_INVALID_ARG, "cache_layer_stride < T*row_elems");
    if (rows_layer_stride < static_cast<long long>(n_rows) * row_elems)
        return fail(CS_ERR_INVALID_ARG, "rows_layer_stride < n_rows*row_elems");
    if (n_layers == 0 || n_rows == 0) return CS_OK;
    if (T == 0) return fail(CS_ERR_INVALID_ARG, "rows to scatter into an empty cache");
    if (cache == nullptr || rows == nullptr || idx == nullptr)
        return fail(CS_ERR_INVALID_ARG, "NULL pointer");
    if (!aligned16(cache) || !aligned16(rows) || (cache_layer_stride * esz) % 16 ||
        (rows_layer_stride * esz) % 16)
        return fail(CS_ERR_INVALID_ARG, "cache, rows and layer strides must be 16-byte aligned");
    {
        const char *c = static_cast<const char *>(cache);
        const char *r = static_cast<const char *>(rows);
        const long long cspan = ((n_layers - 1) * cache_layer_stride + static_cast<long long>(T) * row_elems) * esz;
        const long long rspan = ((n_layers - 1) * rows_layer_stride + static_cast<long long>(n_rows) * row_elems) * esz;
        if (c < r + rspan && r < c + cspan) return fail(CS_ERR_INVALID_ARG, "rows overlap the cache");
        // every warp reads its row's index while others write the cache
        if (overlaps(idx, 4ll * n_rows, cache, cspan))
            return fail(CS_ERR_INVALID_ARG, "idx overlaps the cache");
    }
    unsigned int *status = status_word();
    if (status == nullptr) return CS_ERR_CUDA;
    const long long row16 = row_elems * esz / 16;
    const cudaError_t e = launch_scatter(cache, rows, n_layers, T, cache_layer_stride * esz / 16, n_rows,
                                         rows_layer_stride * esz / 16, static_cast<int>(row16), idx,
                                         status, as_stream(stream));
    if (e != cudaSuccess) return cuda_fail(e, "scatter launch");
    return CS_OK;
}

cs_status cs_repair_attention(const void *q, const void *k, const void *v, void *o, float *lse,
                              cs_dtype dtype, int n_layers, int M, int T, int n_q_heads,
                              int n_kv_heads, int head_dim, int64_t kv_layer_stride,
                              const int32_t *qpos, float scale, void *stream) {
    if (dtype != CS_DTYPE_F32 && dtype != CS_DTYPE_BF16) return fail(CS_ERR_INVALID_ARG, "dtype");
    if (n_layers < 0 || M < 0 || T < 0 || n_q_heads <= 0 || n_kv_heads <= 0 || head_dim <= 0)
        return fail(CS_ERR_INVALID_ARG, "negative size or non-positive head count/dim");
    if (head_dim != 128) return fail(CS_ERR_UNSUPPORTED, "head_dim %d (only 128)", head_dim);
    if (n_q_heads % n_kv_heads)
        return fail(CS_ERR_INVALID_ARG, "n_q_heads %d not a multiple of n_kv_heads %d", n_q_heads,
                    n_kv_heads);
    if (n_q_heads / n_kv_heads > 128)
        return fail(CS_ERR_UNSUPPORTED, "more than 128 query heads per kv head");
    if (!std::isfinite(scale)) return fail(CS_ERR_INVALID_ARG, "scale must be finite");
    if (lse != nullptr && (reinterpret_cast<uintptr_t>(lse) & 3u))
        return fail(CS_ERR_INVALID_ARG, "lse must be 4-byte aligned");
    if (kv_layer_stride < static_cast<long long>(T) * n_kv_heads * head_dim)
        return fail(CS_ERR_INVALID_ARG, "kv_layer_stride < T*n_kv_heads*head_dim");
    if (n_layers == 0 || M == 0) return CS_OK;
    if (T == 0) return fail(CS_ERR_INVALID_ARG, "query rows need at least one key (T = 0)");
    if (q == nullptr || k == nullptr || v == nullptr || o == nullptr || qpos == nullptr)
        return fail(CS_ERR_INVALID_ARG, "NULL pointer");
    const long long esz = dtype == CS_DTYPE_BF16 ? 2 : 4;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) ||
        (kv_layer_stride * esz) % 16)
        return fail(CS_ERR_INVALID_ARG, "q, k, v, o must be 16-byte aligned (and the layer stride)");
    if (dtype == CS_DTYPE_BF16 && static_cast<long long>(M) * n_q_heads > 0x7FFFFFFFll)
        return fail(CS_ERR_UNSUPPORTED, "M * n_q_heads too large");
    {
        // o is written while other CTAs still read k and v (each o element is written by
        // the CTA that read the same element of q, so o == q is allowed)
        const long long kv_span =
            ((n_layers - 1) * kv_layer_stride + static_cast<long long>(T) * n_kv_heads * head_dim) * esz;
        const long long o_span = static_cast<long long>(n_layers) * M * n_q_heads * head_dim * esz;
        const char *oc = static_cast<const char *>(o);
        const char *kc = static_cast<const char *>(k);
        const char *vc = static_cast<const char *>(v);
        if ((oc < kc + kv_span && kc < oc + o_span) || (oc < vc + kv_span && vc < oc + o_span))
            return fail(CS_ERR_INVALID_ARG, "o overlaps k or v");
        // lse is written while other CTAs still read k and v, too
        if (lse != nullptr) {
            const long long l_span = 4ll * n_layers * M * n_q_heads;
            const char *lc = reinterpret_cast<const char *>(lse);
            if ((lc < kc + kv_span && kc < lc + l_span) || (lc < vc + kv_span && vc < lc + l_span))
                return fail(CS_ERR_INVALID_ARG, "lse overlaps k or v");
            if (lc < oc + o_span && oc < lc + l_span)
                return fail(CS_ERR_INVALID_ARG, "lse overlaps o");
            if (overlaps(qpos, 4ll * M, lse, l_span))
                return fail(CS_ERR_INVALID_ARG, "qpos overlaps lse");
        }
        // every CTA reads query positions while others write o (and lse)
        if (overlaps(qpos, 4ll * M, o, o_span))
            return fail(CS_ERR_INVALID_ARG, "qpos overlaps o");
    }
    unsigned int *status = status_word();
    if (status == nullptr) return CS_ERR_CUDA;
    AttnArgs a;
    a.q = q;
    a.k = k;
    a.v = v;
    a.o = o;
    a.lse = lse;
    a.n_layers = n_layers;
    a.M = M;
    a.T = T;
    a.hq = n_q_heads;
    a.hkv = n_kv_heads;
    a.kv_layer_stride = kv_layer_stride;
    a.qpos = qpos;
    a.scale = scale;
    a.status = status;
    if (dtype == CS_DTYPE_F32) {
        const cudaError_t e = launch_attn_f32(a, as_stream(stream));
        if (e != cudaSuccess) return cuda_fail(e, "attention launch");
        return CS_OK;
    }
    return launch_attn_tc(a, as_stream(stream));
}

cs_status cs_sync_status(void *stream) {
    unsigned int *status = status_word();
    if (status == nullptr) return CS_ERR_CUDA;
    const cudaStream_t s = as_stream(stream);
    unsigned long long rec = 0;
    {
        // take the record on the device, in `stream`'s order (exchange with 0, so an error
        // recorded concurrently by a kernel on another stream is either taken now or left
        // for the next call), then wait for the stream and read what was taken
        std::lock_guard<std::mutex> lock(g_take_mu);
        cudaError_t e = launch_status_take(status, s);
        if (e != cudaSuccess) return cuda_fail(e, "status take launch");
        e = cudaMemcpyAsync(&rec, status + 2, sizeof(rec), cudaMemcpyDeviceToHost, s);
        if (e != cudaSuccess) return cuda_fail(e, "reading the status record");
        e = cudaStreamSynchronize(s);
        if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    }
    if (rec == 0) return CS_OK;
    const unsigned int code = static_cast<unsigned int>(rec >> 56);
    const unsigned int site = static_cast<unsigned int>((rec >> 48) & 0xFFu);
    const unsigned int detail = static_cast<unsigned int>(rec & 0xFFFFFFFFu);
    const cs_status st = code == 4u ? CS_ERR_TIMEOUT : CS_ERR_DEVICE_ARG;
    return fail(st, "device status %u at site %u (detail %u)", code, site, detail);
}

}  // extern "C"

// ---- diagnostics: a bounded wait that nothing completes -----------------------
namespace cs {
namespace {
__global__ void wait_timeout_kernel(unsigned int *status, unsigned long long limit_ns) {
    __shared__ uint64_t bar;
    __shared__ int abort;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort = 0;
        fence_mbar_init();
    }
    __syncthreads();
    // phase 0 never completes: nobody arrives on the barrier
    mbar_wait_bounded(&bar, 0, &abort, status, kSiteDebugWait, limit_ns);
}
}  // namespace

cudaError_t launch_wait_timeout(unsigned int *status, unsigned int limit_us, cudaStream_t s) {
    wait_timeout_kernel<<<1, 1, 0, s>>>(status, 1000ull * limit_us);
    return cudaGetLastError();
}

namespace {
// Moves the status record (words 0-1) into the take slot (words 2-3) and clears it,
// in one atomic exchange.
__global__ void status_take_kernel(unsigned int *status) {
    unsigned long long *w = reinterpret_cast<unsigned long long *>(status);
    w[1] = atomicExch(&w[0], 0ull);
}
}  // namespace

cudaError_t launch_status_take(unsigned int *status, cudaStream_t s) {
    status_take_kernel<<<1, 1, 0, s>>>(status);
    return cudaGetLastError();
}
}  // namespace cs

extern "C" cs_status cs_debug_wait_timeout(uint32_t limit_us, void *stream) {
    if (limit_us == 0 || limit_us > 10u * 1000u * 1000u)
        return fail(CS_ERR_INVALID_ARG, "limit_us must be in (0, 10 s]");
    unsigned int *status = status_word();
    if (status == nullptr) return CS_ERR_CUDA;
    const cudaError_t e = launch_wait_timeout(status, limit_us, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "wait-timeout launch");
    return CS_OK;
}
