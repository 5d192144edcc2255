// merge.cu -- the parameter server's merge of the large- and small-batch
// workers' pushes into the fp32 master weights (Sec. 3.4 with Eq. 1 and
// momentum), plus the bf16 copy the workers pull next (Sec. 2.3).
//
// One pass over memory: per parameter it reads w, u, g_L, g_S (16 B) and
// writes w, u (8 B) and the bf16 w16 (2 B), 26 B in all.  The kernel is
// HBM-bound; it moves 4 parameters per thread per step with 128-bit loads,
// streaming (evict-first) cache hints, and two steps in flight per thread.
#include <algorithm>
#include <chrono>
#include <thread>

#include "dbl_internal.cuh"

namespace {

struct MergeArgs {
    float* w;
    float* u;
    act_t* w16;
    const float* gL;
    const float* gS;
    int64_t n;
    float lr, mu, fL, fS;
    int order;
    // loss scaling: each push divided by the scale its worker used (NULL: 1), and the whole
    // update skipped when *skip is non-zero (a pushed value was not finite)
    const float* scaleL;
    const float* scaleS;
    const int32_t* skip;
};

// One momentum step per push, in the order the server receives them.
__device__ __forceinline__ void merge_one(float& w, float& u, float gl, float gs, const MergeArgs& a, bool hasL,
                                          bool hasS)
{
    if (a.order == 2) {
        float g = 0.f;
        if (hasL) g = a.fL * gl;
        if (hasS) g = fmaf(a.fS, gs, g);
        u = a.mu * u - a.lr * g;
        w = w + u;
        return;
    }
    const bool lfirst = a.order == 0;
    const bool has1 = lfirst ? hasL : hasS, has2 = lfirst ? hasS : hasL;
    const float g1 = lfirst ? gl : gs, g2 = lfirst ? gs : gl;
    const float f1 = lfirst ? a.fL : a.fS, f2 = lfirst ? a.fS : a.fL;
    if (has1) {
        u = a.mu * u - a.lr * (f1 * g1);
        w = w + u;
    }
    if (has2) {
        u = a.mu * u - a.lr * (f2 * g2);
        w = w + u;
    }
}

__device__ __forceinline__ float4 ld_stream(const float* p) { return __ldcs(reinterpret_cast<const float4*>(p)); }

__global__ void __launch_bounds__(256) ps_merge_kernel(MergeArgs a)
{
    if (a.skip && *a.skip) return;
    const bool hasL = a.gL != nullptr, hasS = a.gS != nullptr;
    // 1/S is exact for the power-of-two scales of dynamic loss scaling; 1 without scaling
    const float invL = a.scaleL ? 1.0f / *a.scaleL : 1.0f, invS = a.scaleS ? 1.0f / *a.scaleS : 1.0f;
    const int64_t n4 = a.n >> 2;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    // two independent float4 groups per iteration keep more loads in flight
    for (; i + stride < n4; i += 2 * stride) {
        float4 w[2], u[2], gl[2] = {}, gs[2] = {};
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            const int64_t e = (i + k * stride) * 4;
            w[k] = ld_stream(a.w + e);
            u[k] = ld_stream(a.u + e);
            if (hasL) gl[k] = ld_stream(a.gL + e);
            if (hasS) gs[k] = ld_stream(a.gS + e);
        }
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            merge_one(w[k].x, u[k].x, gl[k].x * invL, gs[k].x * invS, a, hasL, hasS);
            merge_one(w[k].y, u[k].y, gl[k].y * invL, gs[k].y * invS, a, hasL, hasS);
            merge_one(w[k].z, u[k].z, gl[k].z * invL, gs[k].z * invS, a, hasL, hasS);
            merge_one(w[k].w, u[k].w, gl[k].w * invL, gs[k].w * invS, a, hasL, hasS);
            const int64_t e = (i + k * stride) * 4;
            __stcs(reinterpret_cast<float4*>(a.w + e), w[k]);
            __stcs(reinterpret_cast<float4*>(a.u + e), u[k]);
            if (a.w16) {
                act2_t lo = dbl::act::pack2(w[k].x, w[k].y);
                act2_t hi = dbl::act::pack2(w[k].z, w[k].w);
                uint2 pk;
                pk.x = *reinterpret_cast<uint32_t*>(&lo);
                pk.y = *reinterpret_cast<uint32_t*>(&hi);
                __stcs(reinterpret_cast<uint2*>(a.w16 + e), pk);
            }
        }
    }
    for (; i < n4; i += stride) {
        const int64_t e = i * 4;
        float4 w = ld_stream(a.w + e), u = ld_stream(a.u + e), gl = {}, gs = {};
        if (hasL) gl = ld_stream(a.gL + e);
        if (hasS) gs = ld_stream(a.gS + e);
        merge_one(w.x, u.x, gl.x * invL, gs.x * invS, a, hasL, hasS);
        merge_one(w.y, u.y, gl.y * invL, gs.y * invS, a, hasL, hasS);
        merge_one(w.z, u.z, gl.z * invL, gs.z * invS, a, hasL, hasS);
        merge_one(w.w, u.w, gl.w * invL, gs.w * invS, a, hasL, hasS);
        __stcs(reinterpret_cast<float4*>(a.w + e), w);
        __stcs(reinterpret_cast<float4*>(a.u + e), u);
        if (a.w16) {
            act2_t lo = dbl::act::pack2(w.x, w.y);
            act2_t hi = dbl::act::pack2(w.z, w.w);
            uint2 pk;
            pk.x = *reinterpret_cast<uint32_t*>(&lo);
            pk.y = *reinterpret_cast<uint32_t*>(&hi);
            __stcs(reinterpret_cast<uint2*>(a.w16 + e), pk);
        }
    }
    // scalar tail (n not a multiple of 4)
    const int64_t t = (n4 << 2) + (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t < a.n && t < (n4 << 2) + 4) {
        float w = a.w[t], u = a.u[t];
        merge_one(w, u, hasL ? a.gL[t] * invL : 0.f, hasS ? a.gS[t] * invS : 0.f, a, hasL, hasS);
        a.w[t] = w;
        a.u[t] = u;
        if (a.w16) a.w16[t] = dbl::act::from_f(w);
    }
}

}  // namespace

namespace {

int merge_launch(float* w, float* u, void* w16_out, const float* g_large, const float* g_small, int64_t n,
                 const dbl_merge_params* p, const float* scale_l, const float* scale_s, const int32_t* skip,
                 void* stream)
{
    using namespace dbl;
    if (!w || !u || !p || n < 0) return set_error(DBL_ERR_INVALID, "ps_merge: null w/u/params or n < 0");
    if (!g_large && !g_small) return set_error(DBL_ERR_INVALID, "ps_merge: no push (both gradients NULL)");
    if (p->order < 0 || p->order > 2) return set_error(DBL_ERR_INVALID, "ps_merge: order must be 0, 1 or 2");
    if (!aligned16(w) || !aligned16(u) || (g_large && !aligned16(g_large)) || (g_small && !aligned16(g_small)) ||
        (w16_out && !aligned16(w16_out)))
        return set_error(DBL_ERR_INVALID, "ps_merge: buffers must be 16-byte aligned");
    if (n == 0) return DBL_OK;
    MergeArgs a{w, u, reinterpret_cast<act_t*>(w16_out), g_large, g_small, n, p->lr, p->momentum,
                p->f_large, p->f_small, p->order, scale_l, scale_s, skip};
    const int64_t n4 = n >> 2;
    const int threads = 256;
    int64_t want = (n4 + 2 * threads - 1) / (2 * threads);
    const int64_t cap = (int64_t)sm_count() * 8;  // 8 resident 256-thread CTAs per SM
    int blocks = (int)(want < cap ? (want < 1 ? 1 : want) : cap);
    ps_merge_kernel<<<blocks, threads, 0, as_stream(stream)>>>(a);
    return launch_check("ps_merge launch");
}

// found_inf |= any element of g[0, n) is not finite
__global__ void __launch_bounds__(256) grads_finite_kernel(const float* __restrict__ g, int64_t n,
                                                           int32_t* __restrict__ found_inf)
{
    bool bad = false;
    const int64_t n4 = n >> 2, stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
        const float4 v = __ldcs(reinterpret_cast<const float4*>(g) + i);
        bad |= !(isfinite(v.x) && isfinite(v.y) && isfinite(v.z) && isfinite(v.w));
    }
    const int64_t t = (n4 << 2) + (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (t < n && t < (n4 << 2) + 4) bad |= !isfinite(g[t]);
    if (__syncthreads_or(bad) && threadIdx.x == 0) atomicExch(found_inf, 1);
}

__global__ void loss_scale_update_kernel(dbl_loss_scale* st, int32_t interval)
{
    if (st->found_inf) {
        st->scale *= 0.5f;
        st->good_steps = 0;
        st->skipped += 1;
    } else if (++st->good_steps >= interval) {
        st->scale *= 2.0f;
        st->good_steps = 0;
    }
    st->found_inf = 0;
}

}  // namespace

extern "C" int dbl_ps_dual_batch_merge(float* w, float* u, void* w16_out, const float* g_large, const float* g_small,
                                       int64_t n, const dbl_merge_params* p, void* stream)
{
    return merge_launch(w, u, w16_out, g_large, g_small, n, p, nullptr, nullptr, nullptr, stream);
}

extern "C" int dbl_ps_dual_batch_merge_scaled(float* w, float* u, void* w16_out, const float* g_large,
                                              const float* g_small, int64_t n, const dbl_merge_params* p,
                                              const float* scale_large, const float* scale_small,
                                              const int32_t* found_inf, void* stream)
{
    using namespace dbl;
    if ((g_large && !scale_large) || (g_small && !scale_small) || !found_inf)
        return set_error(DBL_ERR_INVALID, "ps_merge_scaled: each push needs its scale, and found_inf is required");
    return merge_launch(w, u, w16_out, g_large, g_small, n, p, scale_large, scale_small, found_inf, stream);
}

extern "C" int dbl_grads_finite(const float* g, int64_t n, int32_t* found_inf, void* stream)
{
    using namespace dbl;
    if (!g || !found_inf || n < 0 || !aligned16(g)) return set_error(DBL_ERR_INVALID, "grads_finite: bad arguments");
    if (n == 0) return DBL_OK;
    const int64_t want = ((n >> 2) + 255) / 256;
    const int64_t cap = (int64_t)sm_count() * 8;
    const int blocks = (int)std::max<int64_t>(1, std::min(want, cap));
    grads_finite_kernel<<<blocks, 256, 0, as_stream(stream)>>>(g, n, found_inf);
    return launch_check("grads_finite launch");
}

extern "C" int dbl_loss_scale_update(dbl_loss_scale* state, int32_t growth_interval, void* stream)
{
    using namespace dbl;
    if (!state || growth_interval < 1) return set_error(DBL_ERR_INVALID, "loss_scale_update: bad arguments");
    loss_scale_update_kernel<<<1, 1, 0, as_stream(stream)>>>(state, growth_interval);
    return launch_check("loss_scale_update launch");
}

extern "C" int dbl_zero_f32_2d(float* base, int64_t rows, int64_t cols, int64_t ld, void* stream)
{
    using namespace dbl;
    if (!base || rows < 0 || cols < 0 || ld < cols) return set_error(DBL_ERR_INVALID, "zero_f32_2d: bad arguments");
    if (rows == 0 || cols == 0) return DBL_OK;
    return cuda_check(cudaMemset2DAsync(base, (size_t)ld * sizeof(float), 0, (size_t)cols * sizeof(float), (size_t)rows,
                                        as_stream(stream)),
                      "zero_f32_2d");
}

// ----------------------------------------------------------------------------- late and missing pushes
// Under ASP the server applies whatever push arrives and does not wait for a worker that
// has stopped (Sec. 2.4).  On one GPU a worker is a stream, so "has not pushed" is an
// event that has not completed by the server's deadline; dbl_event_wait gives the host
// that deadline.  dbl_hold holds a worker's stream until the host releases it: a push
// delayed as on the paper's network (a straggler), bounded so that it always ends.
namespace {

__device__ __forceinline__ uint64_t global_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__global__ void hold_kernel(const volatile uint32_t* flag, uint64_t timeout_ns, int32_t* status)
{
    const uint64_t t0 = global_ns();
    int32_t rc = DBL_ERR_TIMEOUT;
    // bounded twice: by the timeout, and by an iteration count that takes far longer at
    // the sleep's minimum of 1 us per poll
    for (uint32_t it = 0; it < (1u << 30); ++it) {
        if (*flag) {
            rc = DBL_OK;
            break;
        }
        if (global_ns() - t0 >= timeout_ns) break;
        __nanosleep(1000);
    }
    if (status) *status = rc;
}

}  // namespace

extern "C" int dbl_hold(const uint32_t* flag, double timeout_s, int32_t* status, void* stream)
{
    using namespace dbl;
    if (!flag || (reinterpret_cast<uintptr_t>(flag) & 3)) return set_error(DBL_ERR_INVALID, "hold: flag must be 4-byte aligned");
    if (!(timeout_s > 0.0 && timeout_s <= 10.0)) return set_error(DBL_ERR_INVALID, "hold: timeout must be in (0, 10] s");
    hold_kernel<<<1, 1, 0, as_stream(stream)>>>(flag, (uint64_t)(timeout_s * 1e9), status);
    return launch_check("hold launch");
}

extern "C" int dbl_event_wait(void* event, double timeout_s)
{
    using namespace dbl;
    if (!event || !(timeout_s >= 0.0)) return set_error(DBL_ERR_INVALID, "event_wait: null event or negative timeout");
    const auto t0 = std::chrono::steady_clock::now();
    for (;;) {
        const cudaError_t e = cudaEventQuery(static_cast<cudaEvent_t>(event));
        if (e == cudaSuccess) return DBL_OK;
        if (e != cudaErrorNotReady) return cuda_check(e, "event_wait: cudaEventQuery");
        const double waited = std::chrono::duration<double>(std::chrono::steady_clock::now() - t0).count();
        if (waited >= timeout_s)
            return set_error(DBL_ERR_TIMEOUT, "event_wait: not complete after %.3f s", timeout_s);
        std::this_thread::sleep_for(std::chrono::microseconds(50));
    }
}
