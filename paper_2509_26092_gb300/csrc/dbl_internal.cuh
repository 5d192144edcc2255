// dbl_internal.cuh -- shared internals of libdbl.so: error reporting, argument
// checks and the sm_103a PTX wrappers (mbarrier, TMA, tcgen05/TMEM) the kernels
// are written with.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/dbl.h"
#include "dbl_act.cuh"

// ---------------------------------------------------------------------------- host-side errors
namespace dbl {

int set_error(int code, const char* fmt, ...);  // records the message, returns code
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline int cuda_check(cudaError_t e, const char* what)
{
    if (e == cudaSuccess) return DBL_OK;
    return set_error(DBL_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Counts one kernel launch (see dbl_kernel_launches).
void count_launch();

// Launch-error check after a kernel launch (does not synchronise); every
// launch site calls it exactly once, which is also how launches are counted.
inline int launch_check(const char* what)
{
    count_launch();
    return cuda_check(cudaGetLastError(), what);
}

inline cudaStream_t as_stream(void* s) { return reinterpret_cast<cudaStream_t>(s); }

// Number of SMs of the current device (cached per device).
int sm_count();

// Tensor-map encoders from the driver, fetched through the runtime's
// entry-point query so the library does not link libcuda directly.
typedef CUresult (*PFN_encodeTiled)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                    const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                    CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
typedef CUresult (*PFN_encodeIm2col)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                     const cuuint64_t*, const int*, const int*, cuuint32_t, cuuint32_t,
                                     const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                     CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
PFN_encodeTiled encode_tiled();
PFN_encodeIm2col encode_im2col();
// Unique ID of the calling thread's current CUDA context (cuCtxGetId), 0 if no
// context is current yet.  IDs are never reused within a process, so a context
// destroyed and created again (cudaDeviceReset) gets a new one.
int current_context_id(unsigned long long* id);

// BatchNorm forward finalize (bn.cu): channel sums over count rows -> saved mean and
// 1/sqrt(var + eps), once per channel in fp64.  Launches on st; returns a status.
int bn_fwd_finalize(int64_t count, int C, float eps, const float* sum, const float* sumsq, float* save_mean,
                    float* save_invstd, cudaStream_t st);

}  // namespace dbl

// ---------------------------------------------------------------------------- device helpers
#if defined(__CUDACC__)

namespace dbl {
namespace dev {

// Bounded waits: every spin on an mbarrier gives up after this much
// wall-clock time (ns, %globaltimer), or after this many polls, whichever
// comes first.  A legitimate wait in these kernels lasts microseconds.
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s
constexpr uint32_t kWaitLimitPolls = 1u << 30;

__device__ __forceinline__ uint32_t smem_u32(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Wait until the phase with the given parity has completed.  Returns false
// if the wait gave up (time or poll limit), or if *abort became nonzero
// (another role of the CTA gave up first).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort)
{
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer();
    for (uint32_t i = 0; i < kWaitLimitPolls; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 63u) == 63u) {
            if (*abort) return false;
            if (globaltimer() - t0 > kWaitLimitNs) return false;
        }
    }
    return false;
}

// Wait for a phase on the way out of an aborted CTA: bounded by a short time,
// not by the abort flag.
__device__ __forceinline__ bool mbar_wait_drain(uint64_t* bar, uint32_t parity)
{
    const uint64_t t0 = globaltimer();
    for (uint32_t i = 0; i < kWaitLimitPolls; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 63u) == 63u && globaltimer() - t0 > kWaitLimitNs / 8) return false;
    }
    return false;
}

// Warp-uniform forms for the MMA and TMA issuing warps.  All 32 lanes run
// the same straight-line code: the wait loop lives inside one asm block (no
// lane-dependent C++ control flow around the tcgen05/TMA issue, which would
// otherwise slow the issue rate about threefold), and the single-thread
// operations are issued by the lane that elect.sync picks (the lowest active
// lane, so the same lane every time in a converged warp).
//
// Bounded wait: returns 1 once the phase with the given parity has
// completed, 0 if *abort is (or becomes) nonzero, or if the poll or time
// limit ran out, in which case it sets *abort itself so that every other
// wait of the CTA gives up promptly.  abort points to shared memory.
__device__ __forceinline__ uint32_t mbar_wait_warp(uint64_t* bar, uint32_t parity, volatile int* abort)
{
    uint32_t ok;
    asm volatile(
        "{\n\t"
        ".reg .pred P1, P2;\n\t"
        ".reg .u32 cnt, fl;\n\t"
        ".reg .u64 t0, t1;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 P1, [%1], %2;\n\t"
        "@P1 bra WAIT_END;\n\t"
        "mov.u32 cnt, 0;\n\t"
        "mov.u64 t0, %%globaltimer;\n"
        "WAIT_POLL:\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 P1, [%1], %2;\n\t"
        "@P1 bra WAIT_END;\n\t"
        "add.u32 cnt, cnt, 1;\n\t"
        "and.b32 fl, cnt, 63;\n\t"
        "setp.ne.u32 P2, fl, 0;\n\t"
        "@P2 bra WAIT_POLL;\n\t"
        "setp.ge.u32 P2, cnt, %5;\n\t"
        "@P2 bra WAIT_FAIL;\n\t"
        "ld.volatile.shared.u32 fl, [%3];\n\t"
        "setp.ne.u32 P2, fl, 0;\n\t"
        "@P2 bra WAIT_END;\n\t"
        "mov.u64 t1, %%globaltimer;\n\t"
        "sub.u64 t1, t1, t0;\n\t"
        "setp.lt.u64 P2, t1, %4;\n\t"
        "@P2 bra WAIT_POLL;\n"
        "WAIT_FAIL:\n\t"
        "st.volatile.shared.u32 [%3], 1;\n"
        "WAIT_END:\n\t"
        "selp.u32 %0, 1, 0, P1;\n\t"
        "}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(smem_u32(const_cast<int*>(abort))), "l"(kWaitLimitNs),
          "r"(kWaitLimitPolls)
        : "memory");
    return ok;
}

// Warp-uniform wait on the way out of an aborted CTA: bounded by a short
// time, not by the abort flag.  Returns 1 if the phase completed.
__device__ __forceinline__ uint32_t mbar_drain_warp(uint64_t* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t"
        ".reg .pred P1, P2;\n\t"
        ".reg .u32 cnt;\n\t"
        ".reg .u64 t0, t1;\n\t"
        "mov.u32 cnt, 0;\n\t"
        "mov.u64 t0, %%globaltimer;\n"
        "DRAIN_POLL:\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 P1, [%1], %2;\n\t"
        "@P1 bra DRAIN_END;\n\t"
        "add.u32 cnt, cnt, 1;\n\t"
        "setp.ge.u32 P2, cnt, %4;\n\t"
        "@P2 bra DRAIN_END;\n\t"
        "mov.u64 t1, %%globaltimer;\n\t"
        "sub.u64 t1, t1, t0;\n\t"
        "setp.lt.u64 P2, t1, %3;\n\t"
        "@P2 bra DRAIN_POLL;\n"
        "DRAIN_END:\n\t"
        "selp.u32 %0, 1, 0, P1;\n\t"
        "}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "l"(kWaitLimitNs / 8), "r"(kWaitLimitPolls)
        : "memory");
    return ok;
}

__device__ __forceinline__ void mbar_arrive_expect_tx_elect(uint64_t* bar, uint32_t bytes)
{
    asm volatile(
        "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
        "elect.sync l|E, 0xffffffff;\n\t"
        "@E mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n\t}" ::"r"(smem_u32(bar)),
        "r"(bytes)
        : "memory");
}

// ---------------------------------------------------------------------------- BatchNorm scale / shift
// Per-channel scale and shift of out = y*scale + shift from the saved statistics,
// in fp32 with explicit rounding (no contraction), so that every kernel that applies
// the normalisation (bn.cu, the fused stem max pool in head.cu) and the backward
// pass's ReLU-mask recomputation get the same bits.
__device__ __forceinline__ void bn_scale_shift(float gamma, float beta, float mean, float invstd, float& scale,
                                               float& shift)
{
    scale = __fmul_rn(gamma, invstd);
    shift = __fsub_rn(beta, __fmul_rn(mean, scale));
}

// ---------------------------------------------------------------------------- per-block partial sums
// sum += v with Kahan compensation (comp carries the lost low-order part)
__device__ __forceinline__ void kahan_add(float& sum, float& comp, float v)
{
    const float y = v - comp;
    const float t = sum + y;
    comp = (t - sum) - y;
    sum = t;
}

// Fixed-order column sums of per-block partials part[nparts][2][K] (row p: the two
// sums block p produced for every channel: a convolution epilogue's sum y and sum
// y^2, or the BatchNorm backward's sum g and sum g*xhat).  Called once by all
// threads of a block of kPartialsThreads covering the kPartialsChannels channels
// from kPartialsChannels*blockIdx.x: thread t takes channel t % 8 and stream
// s = t / 8 of 32, and stream s adds the partials s, s+32, ... in fp32 with Kahan
// compensation (sixteen loads in flight).  A warp's load then reads four partial
// rows of eight adjacent channels, four whole 32-byte sectors.  The 32 stream sums
// are added in fp64 by a fixed binary tree over the stream index, lowest bit first
// (shuffles across lanes 8 and 16 apart, then pairs of warps through shared
// memory).  The order depends only on nparts, so the result is the same on every
// launch and GPU.  Returns the channel (for threads t < 8 whose channel is below
// K, else -1) and its two sums.
constexpr int kPartialsThreads = 256;
constexpr int kPartialsChannels = 8;
static_assert(kPartialsThreads == 32 * kPartialsChannels, "32 streams of 8 channels");

__device__ __forceinline__ int partials_colsum(const float* __restrict__ part, int nparts, int K, double& sum0,
                                               double& sum1)
{
    __shared__ double red[2][kPartialsThreads / 32][kPartialsChannels];
    const int cl = threadIdx.x % kPartialsChannels, stream = threadIdx.x / kPartialsChannels;
    const int c = blockIdx.x * kPartialsChannels + cl;
    float s = 0.f, sc = 0.f, q = 0.f, qc = 0.f;
    if (c < K) {
        const int64_t ld = 2 * (int64_t)K;
        for (int t = stream; t < nparts; t += 512) {
            float vs[16], vq[16];
#pragma unroll
            for (int u = 0; u < 16; ++u) {
                const bool in = t + 32 * u < nparts;
                vs[u] = in ? __ldg(part + (int64_t)(t + 32 * u) * ld + c) : 0.f;
                vq[u] = in ? __ldg(part + (int64_t)(t + 32 * u) * ld + K + c) : 0.f;
            }
#pragma unroll
            for (int u = 0; u < 16; ++u)
                if (t + 32 * u < nparts) {
                    kahan_add(s, sc, vs[u]);
                    kahan_add(q, qc, vq[u]);
                }
        }
    }
    double ds = (double)s - (double)sc, dq = (double)q - (double)qc;
    // stream bits 0 and 1 are lane bits 3 and 4
#pragma unroll
    for (int o = 8; o < 32; o <<= 1) {
        ds += __shfl_xor_sync(0xffffffffu, ds, o);
        dq += __shfl_xor_sync(0xffffffffu, dq, o);
    }
    const int w = threadIdx.x / 32;
    if ((threadIdx.x & 31) < kPartialsChannels) {
        red[0][w][cl] = ds;
        red[1][w][cl] = dq;
    }
    __syncthreads();
    if (threadIdx.x < kPartialsChannels) {
        // stream bits 2, 3 and 4 are warp bits 0, 1 and 2
        const double(&a)[8][kPartialsChannels] = red[0];
        const double(&b)[8][kPartialsChannels] = red[1];
        ds = ((a[0][cl] + a[1][cl]) + (a[2][cl] + a[3][cl])) + ((a[4][cl] + a[5][cl]) + (a[6][cl] + a[7][cl]));
        dq = ((b[0][cl] + b[1][cl]) + (b[2][cl] + b[3][cl])) + ((b[4][cl] + b[5][cl]) + (b[6][cl] + b[7][cl]));
    }
    __syncthreads();
    sum0 = ds;
    sum1 = dq;
    return (threadIdx.x < kPartialsChannels && c < K) ? c : -1;
}

// ---------------------------------------------------------------------------- TMA
__device__ __forceinline__ void tma_prefetch_desc(const void* tmap)
{
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}

__device__ __forceinline__ void tma_load_2d(void* dst, const void* tmap, uint64_t* bar, int32_t c0, int32_t c1)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(tmap)), "r"(smem_u32(bar)), "r"(c0), "r"(c1)
        : "memory");
}

__device__ __forceinline__ void tma_load_3d(void* dst, const void* tmap, uint64_t* bar, int32_t c0, int32_t c1,
                                            int32_t c2)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(tmap)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2)
        : "memory");
}

// im2col load of a 4-D NHWC tensor: starting pixel (n, h, w) of the traversal
// and channel offset c, filter-tap offsets (off_w, off_h) inside the
// bounding box encoded in the tensor map.
__device__ __forceinline__ void tma_load_im2col_4d(void* dst, const void* tmap, uint64_t* bar, int32_t c, int32_t w,
                                                   int32_t h, int32_t n, uint16_t off_w, uint16_t off_h)
{
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.im2col.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5, %6}], [%2], {%7, %8};" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(tmap)), "r"(smem_u32(bar)), "r"(c), "r"(w), "r"(h), "r"(n), "h"(off_w),
        "h"(off_h)
        : "memory");
}

// Elected-lane forms of the TMA loads above (whole warp calls, one lane issues).
__device__ __forceinline__ void tma_load_4d_elect(void* dst, const void* tmap, uint64_t* bar, int32_t c0, int32_t c1,
                                                  int32_t c2, int32_t c3)
{
    asm volatile(
        "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
        "elect.sync l|E, 0xffffffff;\n\t"
        "@E cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5, %6}], [%2];\n\t}" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(tmap)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
        : "memory");
}

// ---------------------------------------------------------------------------- CTA pairs (clusters of 2)
// A kernel whose MMAs span a CTA pair (tcgen05 .cta_group::2) uses these forms
// throughout: PTX forbids mixing .cta_group::1 and ::2 tcgen05 instructions in
// one kernel.
__device__ __forceinline__ uint32_t cluster_ctarank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Shared::cluster address of the variable at shared::cta address addr in CTA rank.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

// Every thread of every CTA of the cluster: release this CTA's prior writes
// (barrier inits included), acquire the others'.
__device__ __forceinline__ void cluster_sync_all()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Arrive once on an mbarrier given by its shared::cluster address (possibly in the peer CTA).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr)
{
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// TMA loads whose completion is signalled on the mbarrier at shared::cluster
// address bar.  CG = 2 (.cta_group::2): bar may be in the peer CTA of the pair,
// which is how both CTAs' operand halves complete on the MMA-issuing CTA's barrier.
template <int CG>
__device__ __forceinline__ void tma_load_2d_cg(void* dst, const void* tmap, uint32_t bar, int32_t c0, int32_t c1)
{
    if constexpr (CG == 2)
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            " [%0], [%1, {%3, %4}], [%2];\n\t}" ::"r"(smem_u32(dst)),
            "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(c0), "r"(c1)
            : "memory");
    else
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            " [%0], [%1, {%3, %4}], [%2];\n\t}" ::"r"(smem_u32(dst)),
            "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(c0), "r"(c1)
            : "memory");
}

template <int CG>
__device__ __forceinline__ void tma_load_3d_cg(void* dst, const void* tmap, uint32_t bar, int32_t c0, int32_t c1,
                                               int32_t c2)
{
    if constexpr (CG == 2)
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            " [%0], [%1, {%3, %4, %5}], [%2];\n\t}" ::"r"(smem_u32(dst)),
            "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
            : "memory");
    else
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            " [%0], [%1, {%3, %4, %5}], [%2];\n\t}" ::"r"(smem_u32(dst)),
            "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
            : "memory");
}

template <int CG>
__device__ __forceinline__ void tma_load_4d_cg(void* dst, const void* tmap, uint32_t bar, int32_t c0, int32_t c1,
                                               int32_t c2, int32_t c3)
{
    if constexpr (CG == 2)
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E cp.async.bulk.tensor.4d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            " [%0], [%1, {%3, %4, %5, %6}], [%2];\n\t}" ::"r"(smem_u32(dst)),
            "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
            : "memory");
    else
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            " [%0], [%1, {%3, %4, %5, %6}], [%2];\n\t}" ::"r"(smem_u32(dst)),
            "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
            : "memory");
}

template <int CG>
__device__ __forceinline__ void tma_load_im2col_4d_cg(void* dst, const void* tmap, uint32_t bar, int32_t c, int32_t w,
                                                      int32_t h, int32_t n, uint16_t off_w, uint16_t off_h)
{
    if constexpr (CG == 2)
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E cp.async.bulk.tensor.4d.cta_group::2.shared::cluster.global.im2col.mbarrier::complete_tx::bytes"
            " [%0], [%1, {%3, %4, %5, %6}], [%2], {%7, %8};\n\t}" ::"r"(smem_u32(dst)),
            "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(c), "r"(w), "r"(h), "r"(n), "h"(off_w), "h"(off_h)
            : "memory");
    else
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E cp.async.bulk.tensor.4d.shared::cluster.global.im2col.mbarrier::complete_tx::bytes"
            " [%0], [%1, {%3, %4, %5, %6}], [%2], {%7, %8};\n\t}" ::"r"(smem_u32(dst)),
            "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar), "r"(c), "r"(w), "r"(h), "r"(n), "h"(off_w), "h"(off_h)
            : "memory");
}

// TMEM allocation for CG-CTA MMAs.  CG = 2: one warp of each CTA of the pair
// executes it; both CTAs get the same columns.
template <int CG>
__device__ __forceinline__ void tmem_alloc_cg(uint32_t* slot_smem, uint32_t ncols)
{
    if constexpr (CG == 2)
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot_smem)),
                     "r"(ncols)
                     : "memory");
    else
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot_smem)),
                     "r"(ncols)
                     : "memory");
}

template <int CG>
__device__ __forceinline__ void tmem_relinquish_cg()
{
    if constexpr (CG == 2)
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    else
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

template <int CG>
__device__ __forceinline__ void tmem_dealloc_cg(uint32_t taddr, uint32_t ncols)
{
    if constexpr (CG == 2)
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
    else
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

// Elected-lane MMA.  CG = 2: M = 256 across the pair; A rows 0-127 and B columns
// 0..N/2-1 come from the shared memory of CTA rank 0, A rows 128-255 and B columns
// N/2..N-1 from rank 1, at the same addresses; D rows 0-127 land in rank 0's TMEM,
// rows 128-255 in rank 1's, at the same column address.  Issued by rank 0 only.
template <int CG>
__device__ __forceinline__ void mma_act_elect_cg(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                                  uint32_t accumulate)
{
    if constexpr (CG == 2)
        asm volatile(
            "{\n\t.reg .pred E, P;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "setp.ne.b32 P, %4, 0;\n\t"
            "@E tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, P;\n\t}" ::"r"(d_tmem),
            "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
            : "memory");
    else
        asm volatile(
            "{\n\t.reg .pred E, P;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "setp.ne.b32 P, %4, 0;\n\t"
            "@E tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, P;\n\t}" ::"r"(d_tmem),
            "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
            : "memory");
}

// Four K-steps of two accumulators (8 MMAs, cta_group::1) from one elected lane in
// one asm block: D[d0] and D[d1] (+)= A * B for K-step j = 0..3 with descriptors
// a0 + j*a_step (accumulator 0), a0 + a1_off + j*a_step (accumulator 1) and
// b0 + j*b_step (all in descriptor units of 16 bytes).  K-step 0 accumulates only
// if acc0 != 0; K-steps 1..3 always accumulate.  Keeping the whole group inside
// one asm block (no per-MMA elect or predicate set-up in between) is what lets
// N = 64 MMAs, which the tensor pipe finishes in 48 cycles, issue back to back.
__device__ __forceinline__ void mma_act_x8_elect(uint32_t d0, uint32_t d1, uint64_t a0, uint64_t a1_off,
                                                  uint64_t a_step, uint64_t b0, uint64_t b_step, uint32_t idesc,
                                                  uint32_t acc0)
{
    asm volatile(
        "{\n\t.reg .pred E, P, T;\n\t.reg .b32 l;\n\t.reg .b64 a, c, b;\n\t"
        "elect.sync l|E, 0xffffffff;\n\t"
        "setp.ne.b32 P, %8, 0;\n\t"
        "setp.eq.b32 T, 0, 0;\n\t"
        "add.s64 c, %2, %3;\n\t"
        "@E tcgen05.mma.cta_group::1.kind::f16 [%0], %2, %5, %7, P;\n\t"
        "@E tcgen05.mma.cta_group::1.kind::f16 [%1], c, %5, %7, P;\n\t"
        "add.s64 a, %2, %4;\n\tadd.s64 c, c, %4;\n\tadd.s64 b, %5, %6;\n\t"
        "@E tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %7, T;\n\t"
        "@E tcgen05.mma.cta_group::1.kind::f16 [%1], c, b, %7, T;\n\t"
        "add.s64 a, a, %4;\n\tadd.s64 c, c, %4;\n\tadd.s64 b, b, %6;\n\t"
        "@E tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %7, T;\n\t"
        "@E tcgen05.mma.cta_group::1.kind::f16 [%1], c, b, %7, T;\n\t"
        "add.s64 a, a, %4;\n\tadd.s64 c, c, %4;\n\tadd.s64 b, b, %6;\n\t"
        "@E tcgen05.mma.cta_group::1.kind::f16 [%0], a, b, %7, T;\n\t"
        "@E tcgen05.mma.cta_group::1.kind::f16 [%1], c, b, %7, T;\n\t}" ::"r"(d0),
        "r"(d1), "l"(a0), "l"(a1_off), "l"(a_step), "l"(b0), "l"(b_step), "r"(idesc), "r"(acc0)
        : "memory");
}

// mma_act_x8_elect for CG-CTA MMAs (CG = 2: M = 256 across the pair, issued by rank 0,
// A and B halves at the same shared-memory addresses in both CTAs, as in mma_act_elect_cg).
template <int CG>
__device__ __forceinline__ void mma_act_x8_elect_cg(uint32_t d0, uint32_t d1, uint64_t a0, uint64_t a1_off,
                                                     uint64_t a_step, uint64_t b0, uint64_t b_step, uint32_t idesc,
                                                     uint32_t acc0)
{
    if constexpr (CG == 2)
        asm volatile(
            "{\n\t.reg .pred E, P, T;\n\t.reg .b32 l;\n\t.reg .b64 a, c, b;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "setp.ne.b32 P, %8, 0;\n\t"
            "setp.eq.b32 T, 0, 0;\n\t"
            "add.s64 c, %2, %3;\n\t"
            "@E tcgen05.mma.cta_group::2.kind::f16 [%0], %2, %5, %7, P;\n\t"
            "@E tcgen05.mma.cta_group::2.kind::f16 [%1], c, %5, %7, P;\n\t"
            "add.s64 a, %2, %4;\n\tadd.s64 c, c, %4;\n\tadd.s64 b, %5, %6;\n\t"
            "@E tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %7, T;\n\t"
            "@E tcgen05.mma.cta_group::2.kind::f16 [%1], c, b, %7, T;\n\t"
            "add.s64 a, a, %4;\n\tadd.s64 c, c, %4;\n\tadd.s64 b, b, %6;\n\t"
            "@E tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %7, T;\n\t"
            "@E tcgen05.mma.cta_group::2.kind::f16 [%1], c, b, %7, T;\n\t"
            "add.s64 a, a, %4;\n\tadd.s64 c, c, %4;\n\tadd.s64 b, b, %6;\n\t"
            "@E tcgen05.mma.cta_group::2.kind::f16 [%0], a, b, %7, T;\n\t"
            "@E tcgen05.mma.cta_group::2.kind::f16 [%1], c, b, %7, T;\n\t}" ::"r"(d0),
            "r"(d1), "l"(a0), "l"(a1_off), "l"(a_step), "l"(b0), "l"(b_step), "r"(idesc), "r"(acc0)
            : "memory");
    else
        mma_act_x8_elect(d0, d1, a0, a1_off, a_step, b0, b_step, idesc, acc0);
}

// Elected-lane commit: arrive once on the mbarrier at shared::cta offset bar
// when the MMAs issued so far complete.  CG = 2: the arrival goes to the
// barrier at that offset in every CTA of cta_mask (bit r = rank r).
template <int CG>
__device__ __forceinline__ void mma_commit_elect_cg(uint64_t* bar, uint16_t cta_mask)
{
    if constexpr (CG == 2)
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;\n\t}" ::
                "r"(smem_u32(bar)),
            "h"(cta_mask)
            : "memory");
    else
        asm volatile(
            "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
            "elect.sync l|E, 0xffffffff;\n\t"
            "@E tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(smem_u32(bar))
            : "memory");
}

// ---------------------------------------------------------------------------- tcgen05 / TMEM
__device__ __forceinline__ void tmem_alloc(uint32_t* slot_smem, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot_smem)),
                 "r"(ncols)
                 : "memory");
}

__device__ __forceinline__ void tmem_relinquish()
{
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D[tmem] (+)= A[smem desc] * B[smem desc]^T, kind::f16 (16-bit inputs of the storage format, fp32 accumulate).
__device__ __forceinline__ void mma_act(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive once on the mbarrier when all previously issued MMAs of this thread complete.
__device__ __forceinline__ void mma_commit(uint64_t* bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}

// Elected-lane forms: the whole warp calls, one lane issues.  The commit
// tracks the MMAs issued by the elected lane, which is the same lane that
// mma_act_elect uses in a converged warp.
__device__ __forceinline__ void mma_act_elect(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                               uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred E, P;\n\t.reg .b32 l;\n\t"
        "elect.sync l|E, 0xffffffff;\n\t"
        "setp.ne.b32 P, %4, 0;\n\t"
        "@E tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, P;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit_elect(uint64_t* bar)
{
    asm volatile(
        "{\n\t.reg .pred E;\n\t.reg .b32 l;\n\t"
        "elect.sync l|E, 0xffffffff;\n\t"
        "@E tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n\t}" ::"r"(smem_u32(bar))
        : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns: thread i of the warp gets lane
// (base lane + i), columns col..col+31.
__device__ __forceinline__ void tmem_ld_32x32b_x32(uint32_t taddr, uint32_t (&r)[32])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
}

__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// Wait for this thread's outstanding tcgen05.ld; r (the destination of one of them)
// is passed through the wait so that the compiler reads it only afterwards.  With
// it a thread can keep the next chunk's load in flight while it works on this one.
__device__ __forceinline__ void tmem_ld_wait_regs(uint32_t (&r)[32])
{
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                   "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                   "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                   "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                   "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
                 :
                 : "memory");
}

// ---------------------------------------------------------------------------- UMMA descriptors
// Shared-memory matrix descriptor (tcgen05): start address, leading and
// stride byte offsets (all >> 4), descriptor version 1 at bit 46, swizzle
// mode at bits 61-63 (0 none, 2 = 128-byte swizzle).
enum : uint32_t { kSwizzleNone = 0, kSwizzle128B = 2 };

__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo_bytes, uint32_t sbo_bytes,
                                              uint32_t swizzle)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo_bytes >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo_bytes >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)(swizzle & 7u) << 61;
    return d;
}

// Programmatic dependent launch: a kernel launched with programmatic stream serialization may
// start while the kernel before it on the stream is still running; this waits (once per
// thread) until that kernel has completed and its memory operations are visible.  Without the
// launch attribute it returns at once.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Lets the next kernel on the stream (if launched with programmatic stream serialization) be
// scheduled once every CTA of this one has issued this or exited; it still waits for this
// kernel's completion before touching memory.
__device__ __forceinline__ void grid_dependency_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

// Instruction descriptor, kind::f16 with A and B both in the storage format (bf16, or f16 in the
// fp16 build: one MMA never mixes the two) and fp32 D.
// a_mn / b_mn: 1 if that operand is MN-major (transposed) in shared memory.
__host__ __device__ constexpr uint32_t idesc_act(uint32_t M, uint32_t N, uint32_t a_mn, uint32_t b_mn)
{
    return (1u << 4)            // D: fp32
           | (dbl::act::kMmaFormat << 7)    // A: bf16 (1) or f16 (0), the storage format
           | (dbl::act::kMmaFormat << 10)   // B: the same format as A
           | (a_mn << 15) | (b_mn << 16) | ((N >> 3) << 17) | ((M >> 4) << 24);
}

}  // namespace dev
}  // namespace dbl

#endif  // __CUDACC__
