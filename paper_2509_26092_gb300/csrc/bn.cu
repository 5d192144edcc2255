// bn.cu -- training-mode BatchNorm + residual + ReLU, forward and backward,
// for the ResNet-18 of Sec. 5.1.1.  All kernels are HBM-bound streaming
// passes over [count, C] bf16 tensors with 16-byte (8-channel) vectors.
//
// Forward (one pass, 6 B/element with a residual): the batch statistics come
// from the convolution epilogue (or dbl_bn_stats); every CTA turns them into
// per-channel scale/shift in shared memory, then
//     out = ReLU(y*scale + shift [+ res]).
// Backward (two passes): a reduce pass of sum(g) and sum(g*xhat) per channel
// into per-CTA partials, a tiny fixed-order finalize, and an apply pass
//     dy = gamma*invstd*(g - sum(g)/count - xhat*sum(g*xhat)/count).
#include <mutex>

#include "dbl_internal.cuh"

namespace {

using dbl::dev::bn_scale_shift;

constexpr int kThreads = 256;
constexpr int kMaxC = 2048;
constexpr int kUnroll = 2;  // rows per thread whose loads are in flight together
constexpr int kBlocksPerSM = 4;     // forward apply: 256-thread CTAs resident per SM (64 registers per thread)
constexpr int kBwdBlocksPerSM = 3;  // backward apply pass (85 registers per thread)
constexpr int kReduceBlocksPerSM = 2;  // backward reduce pass: four rows' loads in flight per thread
constexpr int kReduceUnroll = 4;

__device__ __forceinline__ void unpack8(const uint4& v, float (&f)[8])
{
    const act2_t* h = reinterpret_cast<const act2_t*>(&v);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 t = dbl::act::unpack2(h[k]);
        f[2 * k] = t.x;
        f[2 * k + 1] = t.y;
    }
}

__device__ __forceinline__ uint4 pack8(const float (&f)[8])
{
    uint4 v;
    act2_t* h = reinterpret_cast<act2_t*>(&v);
#pragma unroll
    for (int k = 0; k < 4; ++k) h[k] = dbl::act::pack2(f[2 * k], f[2 * k + 1]);
    return v;
}

// ----------------------------------------------------------------------------- statistics
__global__ void __launch_bounds__(kThreads) bn_stats_kernel(const act_t* __restrict__ y, int64_t count, int C,
                                                            float* __restrict__ sum, float* __restrict__ sumsq)
{
    const int groups = C / 8;
    const int g = threadIdx.x % groups;
    const int rstep = kThreads / groups;
    float s[8] = {}, q[8] = {};
    for (int64_t r = (int64_t)blockIdx.x * rstep + threadIdx.x / groups; r < count; r += (int64_t)gridDim.x * rstep) {
        float f[8];
        unpack8(__ldg(reinterpret_cast<const uint4*>(y + r * C) + g), f);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            s[k] += f[k];
            q[k] = fmaf(f[k], f[k], q[k]);
        }
    }
    __shared__ float red[kThreads][17];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        red[threadIdx.x][k] = s[k];
        red[threadIdx.x][8 + k] = q[k];
    }
    __syncthreads();
    if (threadIdx.x < groups) {
        float ts[8] = {}, tq[8] = {};
        for (int t = threadIdx.x; t < rstep * groups; t += groups)
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                ts[k] += red[t][k];
                tq[k] += red[t][8 + k];
            }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            atomicAdd(sum + 8 * threadIdx.x + k, ts[k]);
            atomicAdd(sumsq + 8 * threadIdx.x + k, tq[k]);
        }
    }
}

// ----------------------------------------------------------------------------- forward apply
// Batch statistics -> saved mean and 1/std, once per channel (fp64: the
// variance is E[y^2] - E[y]^2 of sums over up to 10^8 rows).  inv_n = 1/count is
// divided on the host (the same correctly rounded value; an fp64 division on the
// device is a long chain of the GPU's slow fp64 operations).
__global__ void bn_fwd_finalize_kernel(double inv_n, int C, float eps, const float* __restrict__ sum,
                                       const float* __restrict__ sumsq, float* __restrict__ save_mean,
                                       float* __restrict__ save_invstd)
{
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= C) return;
    const double mean = (double)sum[c] * inv_n;
    double var = (double)sumsq[c] * inv_n - mean * mean;
    if (var < 0.0) var = 0.0;
    save_mean[c] = (float)mean;
    save_invstd[c] = (float)rsqrt(var + (double)eps);  // one fp64 sequence instead of a root and a division
}


// The same finalize from a convolution's per-CTA partials part[nparts][2][C]: the
// fixed-order partial sums (partials_colsum, rounded to fp32 as dbl_conv_fwd stores
// them), then mean and 1/std exactly as above.
__global__ void __launch_bounds__(dbl::dev::kPartialsThreads) bn_fwd_finalize_parts_kernel(double inv_n, int C, float eps,
                                                                    const float* __restrict__ part, int nparts,
                                                                    float* __restrict__ save_mean,
                                                                    float* __restrict__ save_invstd)
{
    double ds, dq;
    const int c = dbl::dev::partials_colsum(part, nparts, C, ds, dq);
    if (c < 0) return;
    const float sum = (float)ds, sumsq = (float)dq;
    const double mean = (double)sum * inv_n;
    double var = (double)sumsq * inv_n - mean * mean;
    if (var < 0.0) var = 0.0;
    save_mean[c] = (float)mean;
    save_invstd[c] = (float)rsqrt(var + (double)eps);  // one fp64 sequence instead of a root and a division
}

// Thread t of a CTA owns channel group g = t % (C/8) (8 channels, one 16-byte
// vector) and visits rows t / (C/8), + rows-per-CTA-step, ...; a warp covers
// consecutive vectors of consecutive rows, so every access is coalesced, and the
// channel's scale and shift stay in registers.
__global__ void __launch_bounds__(kThreads, kBlocksPerSM)
    bn_apply_kernel(const act_t* __restrict__ y, const act_t* __restrict__ res,
                    act_t* __restrict__ out, int count, int C, int relu, const float* __restrict__ gamma,
                    const float* __restrict__ beta, const float* __restrict__ mean, const float* __restrict__ invstd)
{
    dbl::dev::grid_dependency_trigger();  // a convolution launched next may start its set-up
    const int groups = C / 8;
    const int g = threadIdx.x % groups;
    const int rstep = kThreads / groups;
    float sc[8], sh[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const int c = 8 * g + k;
        bn_scale_shift(gamma[c], beta[c], mean[c], invstd[c], sc[k], sh[k]);
    }
    const int step = gridDim.x * rstep;
    auto emit = [&](const uint4& yv, const uint4& rv, int v) {
        float f[8], rr[8];
        unpack8(yv, f);
        unpack8(rv, rr);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const float o = __fadd_rn(__fmaf_rn(f[k], sc[k], sh[k]), rr[k]);
            f[k] = (relu && !(o > 0.f)) ? 0.f : o;
        }
        reinterpret_cast<uint4*>(out)[v] = pack8(f);
    };
    const uint4 zero = make_uint4(0, 0, 0, 0);  // bf16 +0 in every lane
    int r = blockIdx.x * rstep + threadIdx.x / groups;
    for (; r + (kUnroll - 1) * step < count; r += kUnroll * step) {
        uint4 yv[kUnroll], rv[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const int v = (r + u * step) * groups + g;
            yv[u] = __ldcs(reinterpret_cast<const uint4*>(y) + v);
            rv[u] = res ? __ldcs(reinterpret_cast<const uint4*>(res) + v) : zero;
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) emit(yv[u], rv[u], (r + u * step) * groups + g);
    }
    for (; r < count; r += step) {
        const int v = r * groups + g;
        emit(__ldcs(reinterpret_cast<const uint4*>(y) + v), res ? __ldcs(reinterpret_cast<const uint4*>(res) + v) : zero,
             v);
    }
}

// ----------------------------------------------------------------------------- backward
// Where the ReLU mask comes from: none (no ReLU), the stored output (out > 0),
// or, when there is no stored output (a BatchNorm without a residual), y,
// recomputed exactly as the forward pass decided it: y*scale + shift > 0 with
// the same fp32 operations.
enum MaskMode : int { kMaskNone = 0, kMaskOut = 1, kMaskY = 2 };

// The raw 16-byte vectors behind one 8-channel group of g = (dout [+ dout2]) * [out > 0]
// and of the BatchNorm input y; loaded together so that several rows' loads are in flight.
struct Vec8 {
    uint4 d, d2, o, y;
};

template <int MASK>
__device__ __forceinline__ void load_g_raw(const act_t* dout, const act_t* dout2,
                                           const act_t* out, const act_t* y, int v, Vec8& g, Vec8& yv)
{
    g.d = __ldcs(reinterpret_cast<const uint4*>(dout) + v);
    g.d2 = dout2 ? __ldcs(reinterpret_cast<const uint4*>(dout2) + v) : make_uint4(0, 0, 0, 0);
    g.o = MASK == kMaskOut ? __ldcs(reinterpret_cast<const uint4*>(out) + v) : make_uint4(0, 0, 0, 0);
    yv.y = __ldcs(reinterpret_cast<const uint4*>(y) + v);
}

template <int MASK>
struct ReluMask {
    float sc[MASK == kMaskY ? 8 : 1], sh[MASK == kMaskY ? 8 : 1];

    __device__ __forceinline__ void init(const float* gamma, const float* beta, const float* mean, const float* invstd,
                                         int g)
    {
        if constexpr (MASK == kMaskY) {
#pragma unroll
            for (int k = 0; k < 8; ++k)
                bn_scale_shift(gamma[8 * g + k], beta[8 * g + k], mean[8 * g + k], invstd[8 * g + k], sc[k], sh[k]);
        }
    }
};

template <int MASK>
__device__ __forceinline__ void combine_g(const Vec8& raw, const float (&y)[8], bool two, const ReluMask<MASK>& m,
                                          float (&g)[8])
{
    unpack8(raw.d, g);
    if (two) {
        float h[8];
        unpack8(raw.d2, h);
#pragma unroll
        for (int k = 0; k < 8; ++k) g[k] += h[k];
    }
    if constexpr (MASK == kMaskY) {
#pragma unroll
        for (int k = 0; k < 8; ++k)
            if (!(__fmaf_rn(y[k], m.sc[k], m.sh[k]) > 0.f)) g[k] = 0.f;
    } else if constexpr (MASK == kMaskOut) {
        float o[8];
        unpack8(raw.o, o);
#pragma unroll
        for (int k = 0; k < 8; ++k)
            if (!(o[k] > 0.f)) g[k] = 0.f;
    }
}

// sg += g, sgc += g*(y - mean)  (the 1/std factor is applied once per partial)
// WRITE_G: also store g (bf16) at vector v of g_out.  The sums are of the fp32 g (the
// dgamma, dbeta outputs keep fp32 accuracy); the apply pass then reads the stored g.
template <int MASK, bool WRITE_G>
__device__ __forceinline__ void accumulate_g(const Vec8& graw, const Vec8& yraw, bool two, const ReluMask<MASK>& relu,
                                             const float (&mu)[8], float (&sg)[8], float (&sgc)[8],
                                             act_t* g_out, int v)
{
    float gg[8], yy[8];
    unpack8(yraw.y, yy);
    combine_g(graw, yy, two, relu, gg);
    if constexpr (WRITE_G) __stcs(reinterpret_cast<uint4*>(g_out) + v, pack8(gg));
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        sg[k] += gg[k];
        sgc[k] = fmaf(gg[k], yy[k] - mu[k], sgc[k]);
    }
}

// Partial blk reduces the row chunks blk, blk + nblk, blk + 2*nblk, ... (a chunk
// is the kThreads/(C/8) rows one CTA covers in one step) into partial[blk][0..C)
// (sum g) and partial[blk][C..2C) (sum g*xhat); CTA b computes partials b,
// b + gridDim.x, ....  Interleaved chunks keep all CTAs streaming through the same
// region of the tensors, and each partial adds its rows in a fixed order, so the
// result does not depend on the grid.
template <int MASK, bool WRITE_G>
__global__ void __launch_bounds__(kThreads, kReduceBlocksPerSM)
    bn_bwd_reduce_kernel(const act_t* __restrict__ dout, const act_t* __restrict__ dout2,
                         const act_t* __restrict__ out, const act_t* __restrict__ y, int count,
                         int C, const float* __restrict__ gamma, const float* __restrict__ beta,
                         const float* __restrict__ mean, const float* __restrict__ invstd, int nblk,
                         float* __restrict__ partial, act_t* __restrict__ g_out)
{
    const int groups = C / 8;
    const int g = threadIdx.x % groups;
    const int rstep = kThreads / groups;
    ReluMask<MASK> rm;
    rm.init(gamma, beta, mean, invstd, g);
    float mu[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) mu[k] = mean[8 * g + k];
    __shared__ float red[kThreads][17];
    const int cstep = nblk * rstep;  // rows from one chunk of a partial to its next
    constexpr int U = kReduceUnroll;  // chunks whose loads are in flight together
    for (int blk = blockIdx.x; blk < nblk; blk += gridDim.x) {
    float sg[8] = {}, sgx[8] = {};
    int r = blk * rstep + threadIdx.x / groups;
    for (; r + (U - 1) * cstep < count; r += U * cstep) {
        Vec8 gg[U], yy[U];
#pragma unroll
        for (int u = 0; u < U; ++u) load_g_raw<MASK>(dout, dout2, out, y, (r + u * cstep) * groups + g, gg[u], yy[u]);
#pragma unroll
        for (int u = 0; u < U; ++u)
            accumulate_g<MASK, WRITE_G>(gg[u], yy[u], dout2 != nullptr, rm, mu, sg, sgx, g_out,
                                        (r + u * cstep) * groups + g);
    }
    for (; r < count; r += cstep) {
        Vec8 gg, yy;
        load_g_raw<MASK>(dout, dout2, out, y, r * groups + g, gg, yy);
        accumulate_g<MASK, WRITE_G>(gg, yy, dout2 != nullptr, rm, mu, sg, sgx, g_out, r * groups + g);
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        red[threadIdx.x][k] = sg[k];
        red[threadIdx.x][8 + k] = sgx[k];
    }
    __syncthreads();
    if (threadIdx.x < groups) {
        float ts[8] = {}, tx[8] = {};
        for (int t = threadIdx.x; t < rstep * groups; t += groups)
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                ts[k] += red[t][k];
                tx[k] += red[t][8 + k];
            }
        float* p = partial + (int64_t)blk * 2 * C;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            p[8 * threadIdx.x + k] = ts[k];
            p[C + 8 * threadIdx.x + k] = tx[k] * invstd[8 * threadIdx.x + k];  // sum g*(y-mean) -> sum g*xhat
        }
    }
    __syncthreads();
    }
}

// Fixed-order sum of the partials [nblk][2][C] (partials_colsum), then dgamma,
// dbeta and the three per-channel coefficients (A, B, C) of the apply pass
// dy = A*g + B*y + C.
__global__ void __launch_bounds__(dbl::dev::kPartialsThreads) bn_bwd_finalize_kernel(
    const float* __restrict__ partial, int nblk, int C, double inv_n, const float* __restrict__ gamma,
    const float* __restrict__ mean, const float* __restrict__ invstd, float* __restrict__ dgamma,
    float* __restrict__ dbeta, float* __restrict__ coef)
{
    double sg, sgx;
    const int c = dbl::dev::partials_colsum(partial, nblk, C, sg, sgx);
    if (c < 0) return;
    dbeta[c] = (float)sg;
    dgamma[c] = (float)sgx;
    // dy = k1*(g - sum(g)/n - xhat*sum(g*xhat)/n), xhat = (y - mean)*invstd, as A*g + B*y + C
    const double k1 = (double)gamma[c] * (double)invstd[c];
    const double k3 = sgx * inv_n;  // inv_n = 1/count, divided on the host
    const double b = -k1 * (double)invstd[c] * k3;
    coef[c] = (float)k1;
    coef[C + c] = (float)b;
    coef[2 * C + c] = (float)(-k1 * (sg * inv_n) - b * (double)mean[c]);
}

template <int MASK>
__global__ void __launch_bounds__(kThreads, kBwdBlocksPerSM)
    bn_bwd_apply_kernel(const act_t* __restrict__ dout, const act_t* __restrict__ dout2,
                        const act_t* __restrict__ out, const act_t* __restrict__ y, int count,
                        int C, const float* __restrict__ gamma, const float* __restrict__ beta,
                        const float* __restrict__ mean, const float* __restrict__ invstd,
                        const float* __restrict__ coef, act_t* __restrict__ dy, act_t* __restrict__ dres)
{
    dbl::dev::grid_dependency_trigger();  // a convolution launched next may start its set-up
    const int groups = C / 8;
    const int g = threadIdx.x % groups;
    const int rstep = kThreads / groups;
    ReluMask<MASK> rm;
    rm.init(gamma, beta, mean, invstd, g);
    float ca[8], cb[8], cc[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const int c = 8 * g + k;
        ca[k] = coef[c];
        cb[k] = coef[C + c];
        cc[k] = coef[2 * C + c];
    }
    const int step = gridDim.x * rstep;
    auto emit = [&](const Vec8& graw, const Vec8& yraw, int v) {
        float gg[8], yy[8], d[8];
        unpack8(yraw.y, yy);
        combine_g(graw, yy, dout2 != nullptr, rm, gg);
#pragma unroll
        for (int k = 0; k < 8; ++k) d[k] = fmaf(ca[k], gg[k], fmaf(cb[k], yy[k], cc[k]));
        __stcs(reinterpret_cast<uint4*>(dy) + v, pack8(d));
        if (dres) __stcs(reinterpret_cast<uint4*>(dres) + v, pack8(gg));
    };
    int r = blockIdx.x * rstep + threadIdx.x / groups;
    for (; r + (kUnroll - 1) * step < count; r += kUnroll * step) {
        Vec8 gg[kUnroll], yy[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) load_g_raw<MASK>(dout, dout2, out, y, (r + u * step) * groups + g, gg[u], yy[u]);
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) emit(gg[u], yy[u], (r + u * step) * groups + g);
    }
    for (; r < count; r += step) {
        Vec8 gg, yy;
        load_g_raw<MASK>(dout, dout2, out, y, r * groups + g, gg, yy);
        emit(gg, yy, r * groups + g);
    }
}

int bn_grid(int64_t nvec, int per_sm = kBlocksPerSM)
{
    int64_t b = (nvec + kThreads - 1) / kThreads;
    const int64_t cap = (int64_t)dbl::sm_count() * per_sm;
    if (b > cap) b = cap;
    return (int)(b < 1 ? 1 : b);
}

// One wave of CTAs that take the same number of partials each (more partials than
// resident CTAs would leave some of them a second round alone).
int reduce_grid(int64_t nblk)
{
    const int64_t cap = (int64_t)dbl::sm_count() * kReduceBlocksPerSM;
    const int64_t per_cta = (nblk + cap - 1) / cap;
    return (int)((nblk + per_cta - 1) / per_cta);
}

int check_shape(const dbl_bn_shape* s, const char* who)
{
    if (!s || s->count < 0 || s->c <= 0) return dbl::set_error(DBL_ERR_INVALID, "%s: bad shape", who);
    if (s->c % 8 != 0 || s->c > kMaxC || (kThreads % (s->c / 8)) != 0)
        return dbl::set_error(DBL_ERR_UNSUPPORTED, "%s: channel count %d (need a multiple of 8 dividing 2048)", who,
                              s->c);
    // the streaming kernels index 16-byte vectors (and rows, plus one grid step, or the
    // reduce's kReduceUnroll chunk strides of at most 512 partials) in 32 bits
    if (s->count * (s->c / 8) + (int64_t)kThreads * dbl::sm_count() * kBlocksPerSM * kUnroll +
            (int64_t)kThreads * 512 * kReduceUnroll >=
        ((int64_t)1 << 31))
        return dbl::set_error(DBL_ERR_UNSUPPORTED, "%s: %lld x %d elements exceed the 2^31-vector limit", who,
                              (long long)s->count, s->c);
    return DBL_OK;
}

// Backward reduce split: a fixed function of the shape (so the workspace size
// and the summation order do not depend on the device): one partial per 2048
// 8-channel vectors (8 per thread), at most kMaxBwdParts.  The cap is below the
// reduce's resident CTAs on this GPU (two per SM), so a large tensor gets one
// partial per CTA; a cap of 512 gave those CTAs two partials each and the
// finalize twice the partials to add (8 us per call at layer4, batch 512).
constexpr int64_t kMaxBwdParts = 256;
int64_t bwd_blocks(int64_t count, int C)
{
    if (count <= 0 || C <= 0) return 1;
    const int64_t b = (count * (C / 8) + 2047) / 2048;
    return b < 1 ? 1 : b > kMaxBwdParts ? kMaxBwdParts : b;
}

template <int MASK>
int bwd_launch_mask(const dbl_bn_shape* s, const void* dout, const void* dout2, const void* y, const void* out,
                    const float* gamma, const float* beta, const float* mean, const float* invstd, void* dy,
                    void* dresidual, float* dgamma, float* dbeta, float* partial, float* coef, int64_t nblk,
                    cudaStream_t st)
{
    using namespace dbl;
    const int C = s->c;
    auto bd = [](const void* p) { return static_cast<const act_t*>(p); };
    // When the caller wants g (the residual branch's gradient), the reduce pass stores it and the
    // apply pass reads it back instead of re-reading dout, dout2 and out.
    act_t* g_store = static_cast<act_t*>(dresidual);
    if (g_store)
        bn_bwd_reduce_kernel<MASK, true><<<reduce_grid(nblk), kThreads, 0, st>>>(
            bd(dout), bd(dout2), bd(out), bd(y), (int)s->count, C, gamma, beta, mean, invstd, (int)nblk, partial,
            g_store);
    else
        bn_bwd_reduce_kernel<MASK, false><<<reduce_grid(nblk), kThreads, 0, st>>>(
            bd(dout), bd(dout2), bd(out), bd(y), (int)s->count, C, gamma, beta, mean, invstd, (int)nblk, partial,
            nullptr);
    int rc = launch_check("bn_bwd_reduce launch");
    if (rc) return rc;
    bn_bwd_finalize_kernel<<<(C + dbl::dev::kPartialsChannels - 1) / dbl::dev::kPartialsChannels,
                             dbl::dev::kPartialsThreads, 0, st>>>(partial, (int)nblk, C, 1.0 / (double)s->count,
                                                                         gamma, mean, invstd, dgamma, dbeta, coef);
    if ((rc = launch_check("bn_bwd_finalize launch"))) return rc;
    if (g_store)
        bn_bwd_apply_kernel<kMaskNone><<<bn_grid(s->count * C / 8, kBwdBlocksPerSM), kThreads, 0, st>>>(
            g_store, nullptr, nullptr, bd(y), (int)s->count, C, gamma, beta, mean, invstd, coef,
            static_cast<act_t*>(dy), nullptr);
    else
        bn_bwd_apply_kernel<MASK><<<bn_grid(s->count * C / 8, kBwdBlocksPerSM), kThreads, 0, st>>>(
            bd(dout), bd(dout2), bd(out), bd(y), (int)s->count, C, gamma, beta, mean, invstd, coef,
            static_cast<act_t*>(dy), nullptr);
    return launch_check("bn_bwd_apply launch");
}

// The three passes of the backward pass (reduce, fixed-order finalize, apply),
// with the ReLU mask taken from out, recomputed from y (out == NULL), or none.
int bwd_launch(const dbl_bn_shape* s, const void* dout, const void* dout2, const void* y, const void* out,
               const float* gamma, const float* beta, const float* mean, const float* invstd, void* dy, void* dresidual,
               float* dgamma, float* dbeta, float* partial, float* coef, int64_t nblk, cudaStream_t st)
{
    if (!s->relu)
        return bwd_launch_mask<kMaskNone>(s, dout, dout2, y, out, gamma, beta, mean, invstd, dy, dresidual, dgamma,
                                          dbeta, partial, coef, nblk, st);
    if (out)
        return bwd_launch_mask<kMaskOut>(s, dout, dout2, y, out, gamma, beta, mean, invstd, dy, dresidual, dgamma,
                                         dbeta, partial, coef, nblk, st);
    return bwd_launch_mask<kMaskY>(s, dout, dout2, y, out, gamma, beta, mean, invstd, dy, dresidual, dgamma, dbeta,
                                   partial, coef, nblk, st);
}

}  // namespace

namespace dbl {

int bn_fwd_finalize(int64_t count, int C, float eps, const float* sum, const float* sumsq, float* save_mean,
                    float* save_invstd, cudaStream_t st)
{
    bn_fwd_finalize_kernel<<<(C + 127) / 128, 128, 0, st>>>(1.0 / (double)count, C, eps, sum, sumsq, save_mean,
                                                            save_invstd);
    return launch_check("bn_fwd_finalize launch");
}

}  // namespace dbl

extern "C" {

int dbl_bn_stats(const dbl_bn_shape* s, const void* y, float* ch_sum, float* ch_sumsq, void* stream)
{
    using namespace dbl;
    int rc = check_shape(s, "bn_stats");
    if (rc) return rc;
    if (!y || !ch_sum || !ch_sumsq || !aligned16(y)) return set_error(DBL_ERR_INVALID, "bn_stats: bad pointer");
    cudaStream_t st = as_stream(stream);
    if ((rc = cuda_check(cudaMemsetAsync(ch_sum, 0, sizeof(float) * s->c, st), "bn_stats memset"))) return rc;
    if ((rc = cuda_check(cudaMemsetAsync(ch_sumsq, 0, sizeof(float) * s->c, st), "bn_stats memset"))) return rc;
    if (s->count == 0) return DBL_OK;
    bn_stats_kernel<<<bn_grid(s->count * s->c / 8), kThreads, 0, st>>>(static_cast<const act_t*>(y), s->count,
                                                                       s->c, ch_sum, ch_sumsq);
    return launch_check("bn_stats launch");
}

int dbl_bn_relu_fused(const dbl_bn_shape* s, const void* y, const float* ch_sum, const float* ch_sumsq,
                      const float* gamma, const float* beta, const void* residual, void* out, float* save_mean,
                      float* save_invstd, void* stream)
{
    using namespace dbl;
    int rc = check_shape(s, "bn_relu_fused");
    if (rc) return rc;
    if (!y || !out || !ch_sum || !ch_sumsq || !gamma || !beta || !save_mean || !save_invstd)
        return set_error(DBL_ERR_INVALID, "bn_relu_fused: null pointer");
    if (!aligned16(y) || !aligned16(out) || (residual && !aligned16(residual)))
        return set_error(DBL_ERR_INVALID, "bn_relu_fused: tensors must be 16-byte aligned");
    if (s->count == 0) return set_error(DBL_ERR_INVALID, "bn_relu_fused: empty batch has no statistics");
    cudaStream_t st = as_stream(stream);
    if ((rc = bn_fwd_finalize(s->count, s->c, s->eps, ch_sum, ch_sumsq, save_mean, save_invstd, st))) return rc;
    bn_apply_kernel<<<bn_grid(s->count * s->c / 8), kThreads, 0, st>>>(
        static_cast<const act_t*>(y), static_cast<const act_t*>(residual),
        static_cast<act_t*>(out), (int)s->count, s->c, s->relu, gamma, beta, save_mean, save_invstd);
    return launch_check("bn_relu_fused launch");
}

int dbl_bn_relu_fused_parts(const dbl_bn_shape* s, const void* y, const float* parts, int32_t nparts,
                            const float* gamma, const float* beta, const void* residual, void* out, float* save_mean,
                            float* save_invstd, void* stream)
{
    using namespace dbl;
    int rc = check_shape(s, "bn_relu_fused_parts");
    if (rc) return rc;
    if (!y || !out || !parts || !gamma || !beta || !save_mean || !save_invstd)
        return set_error(DBL_ERR_INVALID, "bn_relu_fused_parts: null pointer");
    if (nparts <= 0) return set_error(DBL_ERR_INVALID, "bn_relu_fused_parts: no partials");
    if (!aligned16(y) || !aligned16(out) || (residual && !aligned16(residual)))
        return set_error(DBL_ERR_INVALID, "bn_relu_fused_parts: tensors must be 16-byte aligned");
    if (s->count == 0) return set_error(DBL_ERR_INVALID, "bn_relu_fused_parts: empty batch has no statistics");
    cudaStream_t st = as_stream(stream);
    bn_fwd_finalize_parts_kernel<<<(s->c + dbl::dev::kPartialsChannels - 1) / dbl::dev::kPartialsChannels,
                                   dbl::dev::kPartialsThreads, 0, st>>>(1.0 / (double)s->count, s->c, s->eps, parts,
                                                                   nparts, save_mean, save_invstd);
    if ((rc = launch_check("bn_fwd_finalize_parts launch"))) return rc;
    bn_apply_kernel<<<bn_grid(s->count * s->c / 8), kThreads, 0, st>>>(
        static_cast<const act_t*>(y), static_cast<const act_t*>(residual),
        static_cast<act_t*>(out), (int)s->count, s->c, s->relu, gamma, beta, save_mean, save_invstd);
    return launch_check("bn_relu_fused_parts launch");
}

size_t dbl_bn_workspace_bytes(const dbl_bn_shape* s)
{
    if (!s || s->c <= 0) return 0;
    return sizeof(float) * ((size_t)bwd_blocks(s->count, s->c) * 2 * s->c + 3 * (size_t)s->c);
}

int dbl_bn_relu_fused_bwd(const dbl_bn_shape* s, const void* dout, const void* dout2, const void* y, const void* out,
                          const float* gamma, const float* beta, const float* save_mean, const float* save_invstd, void* dy,
                          void* dresidual, float* dgamma, float* dbeta, void* ws, size_t ws_bytes, void* stream)
{
    using namespace dbl;
    int rc = check_shape(s, "bn_relu_fused_bwd");
    if (rc) return rc;
    if (!dout || !y || !dy || !gamma || !save_mean || !save_invstd || !dgamma || !dbeta || (s->relu && !out && !beta))
        return set_error(DBL_ERR_INVALID, "bn_relu_fused_bwd: null pointer");
    if (!aligned16(dout) || !aligned16(y) || !aligned16(dy) || (dout2 && !aligned16(dout2)) ||
        (out && !aligned16(out)) || (dresidual && !aligned16(dresidual)))
        return set_error(DBL_ERR_INVALID, "bn_relu_fused_bwd: tensors must be 16-byte aligned");
    if (s->count == 0) return set_error(DBL_ERR_INVALID, "bn_relu_fused_bwd: empty batch");
    const size_t need = dbl_bn_workspace_bytes(s);
    if (!ws || ws_bytes < need)
        return set_error(DBL_ERR_WORKSPACE, "bn_relu_fused_bwd: workspace %zu < %zu bytes", ws_bytes, need);
    const int C = s->c;
    const int64_t nblk = bwd_blocks(s->count, s->c);
    float* partial = static_cast<float*>(ws);
    float* coef = partial + nblk * 2 * C;
    cudaStream_t st = as_stream(stream);
    return bwd_launch(s, dout, dout2, y, out, gamma, beta, save_mean, save_invstd, dy, dresidual, dgamma, dbeta,
                      partial, coef, nblk, st);
}

}  // extern "C"

// ----------------------------------------------------------------------------- workspace-free variant
// For callers that cannot pass a workspace (see dbl_bn_relu_fused_bwd_noalloc
// in dbl.h): the per-CTA partials and the per-channel coefficients live in
// one file-scope device array sized for the largest channel count accepted.
namespace {

constexpr int kNoallocMaxBlocks = 512;  // bwd_blocks() never exceeds this
constexpr size_t kNoallocFloats =
    (size_t)kNoallocMaxBlocks * 2 * DBL_BN_NOALLOC_MAX_C + 3 * (size_t)DBL_BN_NOALLOC_MAX_C;

static __device__ __align__(256) float g_bn_noalloc_scratch[kNoallocFloats];

// Device address of the array in the calling thread's current context.  It is
// looked up (cudaGetSymbolAddress) the first time a context calls, and cached
// under that context's unique ID: a context destroyed and created again
// (cudaDeviceReset) loads the library's module again, the array may move, and
// the new ID forces a fresh lookup.  A lookup may load the module, which must
// not happen inside a stream capture, so a first call while `st` is capturing
// is refused.  (In host code the array's name is only a stand-in, never a
// device address.)
float* noalloc_scratch(cudaStream_t st, int* rc)
{
    struct Entry {
        unsigned long long ctx;
        float* ptr;
    };
    static std::mutex mu;
    static Entry cache[64] = {};
    static int used = 0;
    unsigned long long ctx = 0;
    if ((*rc = dbl::current_context_id(&ctx))) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; ctx && i < used; ++i)
        if (cache[i].ctx == ctx) {
            *rc = DBL_OK;
            return cache[i].ptr;
        }
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    cudaError_t e = cudaStreamIsCapturing(st, &cs);
    if (e != cudaSuccess || cs != cudaStreamCaptureStatusNone) {
        (void)cudaGetLastError();
        *rc = dbl::set_error(DBL_ERR_INVALID,
                             "bn_bwd_noalloc: the first call in a CUDA context looks up the static scratch and "
                             "must come before any stream capture; call it once outside capture first");
        return nullptr;
    }
    void* p = nullptr;
    if ((*rc = dbl::cuda_check(cudaGetSymbolAddress(&p, g_bn_noalloc_scratch), "bn_bwd_noalloc: cudaGetSymbolAddress")))
        return nullptr;
    if (!ctx && (*rc = dbl::current_context_id(&ctx))) return nullptr;  // the lookup made the context current
    if (ctx && used < 64) cache[used++] = Entry{ctx, static_cast<float*>(p)};  // beyond 64 contexts: no cache
    *rc = DBL_OK;
    return static_cast<float*>(p);
}

}  // namespace

extern "C" int dbl_bn_relu_fused_bwd_noalloc(const dbl_bn_shape* s, const void* dout, const void* dout2,
                                              const void* y, const void* out, const float* gamma, const float* beta,
                                              const float* save_mean, const float* save_invstd, void* dy,
                                              void* dresidual, float* dgamma, float* dbeta, void* stream)
{
    using namespace dbl;
    int rc = check_shape(s, "bn_relu_fused_bwd_noalloc");
    if (rc) return rc;
    if (s->c > DBL_BN_NOALLOC_MAX_C)
        return set_error(DBL_ERR_UNSUPPORTED,
                         "bn_relu_fused_bwd_noalloc: %d channels exceed the static scratch limit of %d", s->c,
                         DBL_BN_NOALLOC_MAX_C);
    if (!dout || !y || !dy || !gamma || !save_mean || !save_invstd || !dgamma || !dbeta || (s->relu && !out && !beta))
        return set_error(DBL_ERR_INVALID, "bn_relu_fused_bwd_noalloc: null pointer");
    if (!aligned16(dout) || !aligned16(y) || !aligned16(dy) || (dout2 && !aligned16(dout2)) ||
        (out && !aligned16(out)) || (dresidual && !aligned16(dresidual)))
        return set_error(DBL_ERR_INVALID, "bn_relu_fused_bwd_noalloc: tensors must be 16-byte aligned");
    if (s->count == 0) return set_error(DBL_ERR_INVALID, "bn_relu_fused_bwd_noalloc: empty batch");
    const int C = s->c;
    const int64_t nblk = bwd_blocks(s->count, s->c);
    if (nblk > kNoallocMaxBlocks || (size_t)nblk * 2 * C + 3 * (size_t)C > kNoallocFloats)
        return set_error(DBL_ERR_UNSUPPORTED, "bn_relu_fused_bwd_noalloc: shape exceeds the static scratch");
    cudaStream_t st = as_stream(stream);
    float* partial = noalloc_scratch(st, &rc);
    if (rc) return rc;
    float* coef = partial + nblk * 2 * C;  // written by the finalize kernel before the apply kernel reads it
    return bwd_launch(s, dout, dout2, y, out, gamma, beta, save_mean, save_invstd, dy, dresidual, dgamma, dbeta,
                      partial, coef, nblk, st);
}
