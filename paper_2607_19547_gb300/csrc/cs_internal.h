// Host-side declarations shared by the translation units of libchronostitch.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/chronostitch.h"

namespace cs {

// Device status area (one per device, 16-byte aligned, four 32-bit words):
//   words 0-1  the first error recorded since the last take, as one 64-bit record
//              (code << 56 | site << 48 | detail; see report_error), 0 if none
//   words 2-3  where cs_sync_status's take kernel leaves the record it removed
constexpr int kStatusWords = 4;

// Returns the device address of the status area of the current device (looked up
// again whenever the current CUDA context differs from the one it was found in), or
// nullptr on a CUDA error (the detail is recorded for cs_last_error_detail).
unsigned int *status_word();

// Number of SMs of the current device (0 if it cannot be queried).
int sm_count();

// Sets a function attribute of `fn` on the current device, once per (function, device):
// function attributes belong to the device's context, so a process that drives several
// devices sets them on each.  Returns the (first) result.
cudaError_t func_attr_once(const void *fn, cudaFuncAttribute attr, int value);

// Records a detail string for cs_last_error_detail and returns `s`.
cs_status fail(cs_status s, const char *fmt, ...);
cs_status cuda_fail(cudaError_t e, const char *what);

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Launches `kernel` with programmatic stream serialization: it may start while the
// previous kernel in `s` is still running.  A kernel launched this way calls
// pdl_wait() (cs_device.cuh) before it reads global memory that an earlier kernel
// may write, so only its launch and set-up overlap the earlier kernel's tail, and
// pdl_trigger() right after, so the next kernel's CTAs may take SMs as this one's
// finish.  Works inside stream capture.  The bf16 attention is launched normally:
// the wait made each of its CTAs start its first loads later (about 4.5 us per
// step at 4x1024), more than the overlap gained.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// ---- re-base (rebase.cu) ---------------------------------------------------
struct RebaseArgs {
    const void *k_in;
    void *k_out;
    int n_layers;
    long long layer_stride;
    int T;
    int hkv;
    const int *pos_local;
    const int *pos_global;
    unsigned long long turn_step[64];   // theta_i / (2 pi) in units of 2^-64 turns
    unsigned char axis[64];             // sigma(i)
    int in_place;
    // fused score of layer score_layer (every supported head count): when score_out
    // is set, score_out[t - cand0] = Eq. 5 squared of fresh row t - cand0 against
    // the re-based row t, for t in [cand0, cand0 + n_cand)
    const void *fresh;
    long long fresh_stride;             // elements between fresh rows
    float *score_out;
    int score_layer, cand0, n_cand;
};
// Whether launch_rebase computes the fused score itself for these arguments.
bool rebase_fuses_score(const RebaseArgs &a, cs_dtype dt);
cudaError_t launch_rebase(const RebaseArgs &a, cs_dtype dt, cudaStream_t s);

// ---- scatter-back (scatter.cu) -----------------------------------------------
cudaError_t launch_scatter(void *cache, const void *rows, int n_layers, int T, long long cache_stride16,
                           int n_rows, long long rows_stride16, int row16, const int *idx,
                           unsigned int *status, cudaStream_t s);

// ---- score (score.cu) --------------------------------------------------------
cudaError_t launch_score(const void *fresh, const void *cached, cs_dtype dt, int n, int E,
                         long long fresh_stride, long long cached_stride, float *out,
                         cudaStream_t s);

// ---- select (select.cu) ------------------------------------------------------
cudaError_t launch_select(const float *score, int n, int k, int idx_base, int *out,
                          cudaStream_t s);

// ---- attention (attn_f32.cu, attn_tc.cu) -------------------------------------
struct AttnArgs {
    const void *q;
    const void *k;
    const void *v;
    void *o;
    float *lse;
    int n_layers, M, T, hq, hkv;
    long long kv_layer_stride;
    const int *qpos;
    float scale;
    unsigned int *status;
};
cudaError_t launch_attn_f32(const AttnArgs &a, cudaStream_t s);
// Returns CS_OK, or an error status with the detail recorded.
cs_status launch_attn_tc(const AttnArgs &a, cudaStream_t s);

cudaError_t launch_wait_timeout(unsigned int *status, unsigned int limit_us, cudaStream_t s);
// Takes the status record into the take slot and clears it (cs_sync_status).
cudaError_t launch_status_take(unsigned int *status, cudaStream_t s);

}  // namespace cs
