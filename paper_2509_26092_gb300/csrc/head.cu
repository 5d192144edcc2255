// head.cu -- the small layers around the convolutions of ResNet-18
// (Sec. 5.1.1): the ImageNet stem's 3x3/2 max pooling, and the head
// (global average pooling -- Sec. 6 -- a fully connected layer and the
// batch-mean softmax cross-entropy of Eq. 1), forward and backward.
//
// These are a few percent of a step's time: the max pool is a bandwidth
// pass over the stem output, the head works on [n, 512] features.  The FC
// products are done by a small tiled fp32 GEMM on the CUDA cores.
#include <float.h>

#include <algorithm>

#include "dbl_internal.cuh"

namespace {

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

int grid_for(int64_t items, int threads, int per_sm = 8)
{
    int64_t b = (items + threads - 1) / threads;
    const int64_t cap = (int64_t)dbl::sm_count() * per_sm;
    if (b > cap) b = cap;
    return (int)(b < 1 ? 1 : b);
}

// ----------------------------------------------------------------------------- max pool 3x3 / 2, pad 1
__global__ void __launch_bounds__(256) maxpool_fwd_kernel(const act_t* __restrict__ x,
                                                          act_t* __restrict__ y, uint8_t* __restrict__ arg,
                                                          int n, int H, int W, int C, int P, int Q)
{
    // 32-bit index math: the host checks that n*P*Q*C/8 fits
    const unsigned groups = (unsigned)C / 8u;
    const unsigned total = (unsigned)n * P * Q * groups;
    for (unsigned t = blockIdx.x * blockDim.x + threadIdx.x; t < total; t += gridDim.x * blockDim.x) {
        const unsigned g = t % groups;
        unsigned pix = t / groups;
        const int q = (int)(pix % (unsigned)Q);
        pix /= (unsigned)Q;
        const int p = (int)(pix % (unsigned)P);
        const int b = (int)(pix / (unsigned)P);
        float best[8];
        uint8_t bi[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            best[k] = -INFINITY;
            bi[k] = 0;
        }
        for (int r = 0; r < 3; ++r) {
            const int h = 2 * p + r - 1;
            if (h < 0 || h >= H) continue;
            for (int s = 0; s < 3; ++s) {
                const int w = 2 * q + s - 1;
                if (w < 0 || w >= W) continue;
                float f[8];
                unpack8(__ldg(reinterpret_cast<const uint4*>(x + (((int64_t)b * H + h) * W + w) * C) + g), f);
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    if (f[k] > best[k]) {  // strict: the first maximum in (r, s) order wins ties
                        best[k] = f[k];
                        bi[k] = (uint8_t)(r * 3 + s);
                    }
            }
        }
        const int64_t o = (((int64_t)b * P + p) * Q + q) * C + 8 * g;
        *reinterpret_cast<uint4*>(y + o) = pack8(best);
        uint2 packed;
        packed.x = bi[0] | (bi[1] << 8) | (bi[2] << 16) | ((uint32_t)bi[3] << 24);
        packed.y = bi[4] | (bi[5] << 8) | (bi[6] << 16) | ((uint32_t)bi[7] << 24);
        *reinterpret_cast<uint2*>(arg + o) = packed;
    }
}

// The same max pool over the output of a training-mode BatchNorm + ReLU
// (no residual) that is never stored: each input vector is normalised as the
// BatchNorm pass would store it, bf16(relu(y*scale + shift)) with the same
// fp32 operations, and then pooled, so the pooled values and the argmax are
// those of pooling the stored BatchNorm output.
// One pair of channels of one input vector through BatchNorm + ReLU, as
// 16-bit pairs of the storage format: each lane is the rounded y*scale + shift from one
// fp32 fma, then max(., 0) in that format, which maps negatives and NaN to zero like the stored
// pass's relu.  A result may be -0 where that pass stores +0; the pool's
// comparisons treat the two alike and the stored maximum is made +0.
__device__ __forceinline__ uint32_t bn_relu_pair(uint32_t w, float2 sc, float2 sh)
{
    const float2 x = dbl::act::unpack2_u32(w);
    const float o0 = __fmaf_rn(x.x, sc.x, sh.x);
    const float o1 = __fmaf_rn(x.y, sc.y, sh.y);
    uint32_t v;
    asm("cvt.rn." DBL_ACT_X2 ".f32 %0, %1, %2;" : "=r"(v) : "f"(o1), "f"(o0));
    asm("max." DBL_ACT_X2 " %0, %1, %2;" : "=r"(v) : "r"(v), "r"(0u));
    return v;
}

// The taps of a window are visited last to first with a >= comparison, so the
// index left is the first maximum in (r, s) order, as in the plain max pool.
// A thread keeps one channel group g for all its windows (the block size is a
// multiple of C/8), so the per-channel scale and shift are computed once, and
// it walks its windows by a fixed pixel stride with carries instead of
// divisions.
__global__ void __launch_bounds__(256)
    bn_relu_maxpool_fwd_kernel(const act_t* __restrict__ x, const float* __restrict__ gamma,
                               const float* __restrict__ beta, const float* __restrict__ mean,
                               const float* __restrict__ invstd, act_t* __restrict__ y,
                               uint8_t* __restrict__ arg, int n, int H, int W, int C, int P, int Q)
{
    dbl::dev::grid_dependency_trigger();  // a convolution launched next may start its set-up
    const unsigned groups = (unsigned)C / 8u;
    const unsigned per_block = blockDim.x / groups;
    if (threadIdx.x >= per_block * groups) return;
    const unsigned g = threadIdx.x % groups;
    const unsigned npix = (unsigned)n * P * Q;
    unsigned pix = blockIdx.x * per_block + threadIdx.x / groups;
    const unsigned stride = gridDim.x * per_block;
    int q = (int)(pix % (unsigned)Q), p = (int)((pix / (unsigned)Q) % (unsigned)P),
        b = (int)(pix / ((unsigned)Q * P));
    const int step_q = (int)(stride % (unsigned)Q), step_p = (int)((stride / (unsigned)Q) % (unsigned)P),
              step_b = (int)(stride / ((unsigned)Q * P));
    float2 sc[4], sh[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int c0 = 8 * g + 2 * k;
        dbl::dev::bn_scale_shift(gamma[c0], beta[c0], mean[c0], invstd[c0], sc[k].x, sh[k].x);
        dbl::dev::bn_scale_shift(gamma[c0 + 1], beta[c0 + 1], mean[c0 + 1], invstd[c0 + 1], sc[k].y, sh[k].y);
    }
    const int64_t row_vecs = (int64_t)W * groups;  // uint4 vectors per input row
    for (; pix < npix; pix += stride) {
        const uint4* xv = reinterpret_cast<const uint4*>(x) + ((int64_t)b * H + 2 * p - 1) * row_vecs +
                          (int64_t)(2 * q - 1) * groups + g;
        const bool r_ok[3] = {p > 0, true, 2 * p + 1 < H};
        const bool s_ok[3] = {q > 0, true, 2 * q + 1 < W};
        // rows last to first, the next row's loads in flight while one is pooled
        uint32_t best[4] = {0u, 0u, 0u, 0u}, idx[4] = {0u, 0u, 0u, 0u};
        uint4 cur[3], nxt[3];
#pragma unroll
        for (int s = 0; s < 3; ++s) {
            cur[s] = (r_ok[2] && s_ok[s]) ? __ldg(xv + 2 * row_vecs + s * (int64_t)groups) : make_uint4(0u, 0u, 0u, 0u);
            nxt[s] = s_ok[s] ? __ldg(xv + row_vecs + s * (int64_t)groups) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int r = 2; r >= 0; --r) {
            if (r_ok[r]) {
#pragma unroll
                for (int s = 2; s >= 0; --s) {
                    if (!s_ok[s]) continue;
                    const uint32_t tap = (uint32_t)(3 * r + s) * 0x10001u;
                    const uint32_t w[4] = {cur[s].x, cur[s].y, cur[s].z, cur[s].w};
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const uint32_t a = bn_relu_pair(w[k], sc[k], sh[k]);
                        uint32_t ge, m;
                        asm("set.ge.u32." DBL_ACT_X2 " %0, %1, %2;" : "=r"(ge) : "r"(a), "r"(best[k]));
                        asm("max." DBL_ACT_X2 " %0, %1, %2;" : "=r"(m) : "r"(best[k]), "r"(a));
                        best[k] = m;
                        idx[k] = (ge & tap) | (~ge & idx[k]);
                    }
                }
            }
            if (r > 0) {
#pragma unroll
                for (int s = 0; s < 3; ++s) {
                    cur[s] = nxt[s];
                    if (r == 2)
                        nxt[s] = (r_ok[0] && s_ok[s]) ? __ldg(xv + s * (int64_t)groups) : make_uint4(0u, 0u, 0u, 0u);
                }
            }
        }
        uint4 out;
        // +0 for a maximum of zero (a -0 lane is negative as a signed 16-bit value)
        asm("max.s16x2 %0, %1, %2;" : "=r"(out.x) : "r"(best[0]), "r"(0u));
        asm("max.s16x2 %0, %1, %2;" : "=r"(out.y) : "r"(best[1]), "r"(0u));
        asm("max.s16x2 %0, %1, %2;" : "=r"(out.z) : "r"(best[2]), "r"(0u));
        asm("max.s16x2 %0, %1, %2;" : "=r"(out.w) : "r"(best[3]), "r"(0u));
        const int64_t o = (int64_t)pix * C + 8 * g;
        *reinterpret_cast<uint4*>(y + o) = out;
        *reinterpret_cast<uint2*>(arg + o) = make_uint2(__byte_perm(idx[0], idx[1], 0x6420),
                                                         __byte_perm(idx[2], idx[3], 0x6420));
        q += step_q;
        if (q >= Q) {
            q -= Q;
            ++p;
        }
        p += step_p;
        if (p >= P) {
            p -= P;
            ++b;
        }
        b += step_b;
    }
}

// dst[k] += src[k] where byte k of the argmax word pair equals tap (fp32; a
// skipped term leaves dst as it is)
__device__ __forceinline__ void add_if_tap(float (&dst)[8], const float (&src)[8], uint2 a, uint32_t tap)
{
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const uint32_t byte = ((k < 4 ? a.x : a.y) >> (8 * (k & 3))) & 0xffu;
        if (byte == tap) dst[k] += src[k];
    }
}

// Gather form over 2x2 blocks of input pixels: block (i, j) = rows 2i..2i+1,
// cols 2j..2j+1 is covered by windows (i..i+1, j..j+1); window (p, q) reaches
// input (h, w) at tap (h - 2p + 1, w - 2q + 1).  So pixel (2i, 2j) takes tap 4
// of window (i, j); (2i, 2j+1) taps 5 and 3 of windows (i, j), (i, j+1);
// (2i+1, 2j) taps 7 and 1 of (i, j), (i+1, j); (2i+1, 2j+1) taps 8, 6, 2, 0
// of the four.  Each pixel sums its windows in (p, q) order, in fp32 from
// zero.  A thread keeps one channel group and steps through the blocks with
// carries, as in the forward pass.
__global__ void __launch_bounds__(256)
    maxpool_bwd_kernel(const act_t* __restrict__ dy, const act_t* __restrict__ dy2,
                       const uint8_t* __restrict__ arg, act_t* __restrict__ dx, int n, int H, int W, int C,
                       int P, int Q)
{
    const unsigned groups = (unsigned)C / 8u;
    const unsigned per_block = blockDim.x / groups;
    if (threadIdx.x >= per_block * groups) return;
    const unsigned g = threadIdx.x % groups;
    const int BH = (H + 1) / 2, BW = (W + 1) / 2;  // BH == P and BW == Q
    const unsigned nblk = (unsigned)n * BH * BW;
    unsigned blk = blockIdx.x * per_block + threadIdx.x / groups;
    const unsigned stride = gridDim.x * per_block;
    int j = (int)(blk % (unsigned)BW), i = (int)((blk / (unsigned)BW) % (unsigned)BH),
        b = (int)(blk / ((unsigned)BW * BH));
    const int step_j = (int)(stride % (unsigned)BW), step_i = (int)((stride / (unsigned)BW) % (unsigned)BH),
              step_b = (int)(stride / ((unsigned)BW * BH));
    const int64_t win_row = (int64_t)Q * C;
    for (; blk < nblk; blk += stride) {
        const bool ok[4] = {true, j + 1 < Q, i + 1 < P, i + 1 < P && j + 1 < Q};
        const int64_t o = (((int64_t)b * P + i) * Q + j) * C + 8 * g;  // window (i, j)
        uint4 gv[4], gv2[4];
        uint2 av[4];
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            const int64_t ot = o + (t >> 1) * win_row + (t & 1) * (int64_t)C;
            gv[t] = ok[t] ? __ldg(reinterpret_cast<const uint4*>(dy + ot)) : make_uint4(0u, 0u, 0u, 0u);
            gv2[t] = (ok[t] && dy2) ? __ldg(reinterpret_cast<const uint4*>(dy2 + ot)) : make_uint4(0u, 0u, 0u, 0u);
            av[t] = ok[t] ? __ldg(reinterpret_cast<const uint2*>(arg + ot)) : make_uint2(~0u, ~0u);
        }
        const bool h1 = 2 * i + 1 < H, w1 = 2 * j + 1 < W;
        act_t* px = dx + (((int64_t)b * H + 2 * i) * W + 2 * j) * C + 8 * g;
        const int64_t px_row = (int64_t)W * C;
        float acc01[8] = {}, acc10[8] = {}, acc11[8] = {};
        {
            float f[8], f2[8], acc00[8] = {};
            unpack8(gv[0], f);
            if (dy2) {
                unpack8(gv2[0], f2);
#pragma unroll
                for (int k = 0; k < 8; ++k) f[k] += f2[k];
            }
            add_if_tap(acc00, f, av[0], 4);
            add_if_tap(acc01, f, av[0], 5);
            add_if_tap(acc10, f, av[0], 7);
            add_if_tap(acc11, f, av[0], 8);
            *reinterpret_cast<uint4*>(px) = pack8(acc00);
        }
        {
            float f[8], f2[8];
            unpack8(gv[1], f);
            if (dy2) {
                unpack8(gv2[1], f2);
#pragma unroll
                for (int k = 0; k < 8; ++k) f[k] += f2[k];
            }
            add_if_tap(acc01, f, av[1], 3);
            add_if_tap(acc11, f, av[1], 6);
            if (w1) *reinterpret_cast<uint4*>(px + C) = pack8(acc01);
        }
        {
            float f[8], f2[8];
            unpack8(gv[2], f);
            if (dy2) {
                unpack8(gv2[2], f2);
#pragma unroll
                for (int k = 0; k < 8; ++k) f[k] += f2[k];
            }
            add_if_tap(acc10, f, av[2], 1);
            add_if_tap(acc11, f, av[2], 2);
            if (h1) *reinterpret_cast<uint4*>(px + px_row) = pack8(acc10);
        }
        {
            float f[8], f2[8];
            unpack8(gv[3], f);
            if (dy2) {
                unpack8(gv2[3], f2);
#pragma unroll
                for (int k = 0; k < 8; ++k) f[k] += f2[k];
            }
            add_if_tap(acc11, f, av[3], 0);
            if (h1 && w1) *reinterpret_cast<uint4*>(px + px_row + C) = pack8(acc11);
        }
        j += step_j;
        if (j >= BW) {
            j -= BW;
            ++i;
        }
        i += step_i;
        if (i >= BH) {
            i -= BH;
            ++b;
        }
        b += step_b;
    }
}

// ----------------------------------------------------------------------------- dropout
// Dropout of the pooled features before the FC layer (Sec. 4.1: the rate rises with the
// resolution, Tables 7 and 9), inverted: a kept feature is scaled by 1/(1 - d).  The draw is
// the counter-based generator Philox4x64-10 (Salmon et al., SC 2011): ten rounds over a
// 256-bit counter with a 128-bit key; a round takes the full 128-bit products of counter
// words 0 and 2 with the two round multipliers and moves the words to
//   (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2), hi(M0*c0) ^ c3 ^ k1, lo(M0*c0)),
// and the key is advanced by the two Weyl increments between rounds.  Feature c of sample n
// takes word c % 4 of the block at counter (n*C/4 + c/4, step, 0, 0), key (seed, 0), and is
// kept when the word's upper 32 bits are >= thr = floor(d * 2^32).
struct Dropout {
    uint32_t thr;          // 0: no dropout
    float scale;           // 1/(1 - d), rounded to fp32
    uint64_t seed;
    const uint64_t* step;  // device counter, read when the kernel runs
    float* mult;           // [n, C] per-feature multiplier (0 or scale) for the backward pass
};

__device__ __forceinline__ void philox4x64_10(uint64_t c[4], uint64_t k0, uint64_t k1)
{
    constexpr uint64_t kM0 = 0xD2E7470EE14C6C93ull, kM1 = 0xCA5A826395121157ull;
    constexpr uint64_t kW0 = 0x9E3779B97F4A7C15ull, kW1 = 0xBB67AE8584CAA73Bull;
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint64_t p0 = kM0 * c[0], q0 = __umul64hi(kM0, c[0]);
        const uint64_t p1 = kM1 * c[2], q1 = __umul64hi(kM1, c[2]);
        const uint64_t a = q1 ^ c[1] ^ k0, b = q0 ^ c[3] ^ k1;
        c[0] = a;
        c[1] = p1;
        c[2] = b;
        c[3] = p0;
        k0 += kW0;
        k1 += kW1;
    }
}

// keep bits (bit j: feature 4*group + j) of one Philox block
__device__ __forceinline__ unsigned dropout_keep4(uint64_t seed, uint64_t step, uint64_t group, uint32_t thr)
{
    uint64_t c[4] = {group, step, 0, 0};
    philox4x64_10(c, seed, 0);
    unsigned bits = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) bits |= (uint32_t)(c[j] >> 32) >= thr ? 1u << j : 0u;
    return bits;
}

__global__ void __launch_bounds__(256) dropout_mask_kernel(int n, int C, uint32_t thr, uint64_t seed,
                                                           const uint64_t* __restrict__ step, uint8_t* __restrict__ keep)
{
    const int64_t groups = (int64_t)n * (C / 4);
    const uint64_t st = thr ? *step : 0;
    for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < groups; g += (int64_t)gridDim.x * blockDim.x) {
        const unsigned b = thr ? dropout_keep4(seed, st, (uint64_t)g, thr) : 0xFu;
        uchar4 v = make_uchar4(b & 1, (b >> 1) & 1, (b >> 2) & 1, (b >> 3) & 1);
        reinterpret_cast<uchar4*>(keep)[g] = v;
    }
}

// ----------------------------------------------------------------------------- head
// feat[n, c] = mean over hw of x[n, hw, c], then (with dropout) times the feature's multiplier
__global__ void __launch_bounds__(256) avgpool_kernel(const act_t* __restrict__ x, float* __restrict__ feat,
                                                      int n, int hw, int C, Dropout dp)
{
    const int groups = C / 8;
    const int64_t total = (int64_t)n * groups;
    const uint64_t st = dp.thr ? *dp.step : 0;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int g = (int)(t % groups);
        const int b = (int)(t / groups);
        float acc[8] = {};
        for (int i = 0; i < hw; ++i) {
            float f[8];
            unpack8(__ldg(reinterpret_cast<const uint4*>(x + ((int64_t)b * hw + i) * C) + g), f);
#pragma unroll
            for (int k = 0; k < 8; ++k) acc[k] += f[k];
        }
        const float inv = 1.0f / (float)hw;
        if (dp.thr) {
            const uint64_t q = (uint64_t)b * (uint64_t)(C / 4) + 2 * (uint64_t)g;
            const unsigned bits = dropout_keep4(dp.seed, st, q, dp.thr) | dropout_keep4(dp.seed, st, q + 1, dp.thr) << 4;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const float m = (bits >> k) & 1 ? dp.scale : 0.f;
                dp.mult[(int64_t)b * C + 8 * g + k] = m;
                feat[(int64_t)b * C + 8 * g + k] = acc[k] * inv * m;
            }
        } else {
#pragma unroll
            for (int k = 0; k < 8; ++k) feat[(int64_t)b * C + 8 * g + k] = acc[k] * inv;
        }
    }
}

// out[m, n] = sum_k A(m,k) * B(n,k) (+ bias[n]); A(m,k) = A[m*sam + k*sak], B(n,k) = B[n*sbn + k*sbk].
// fp32 on the CUDA cores (the head is fp32 end to end): 64 x 64 output tiles, 16-deep K tiles
// stored K-major in shared memory (double-buffered: the next tile is fetched into registers
// while the current one is multiplied), 4 x 4 outputs per thread from float4 reads.  The
// reduction is cut into gridDim.z fixed chunks of kchunk (a function of the shape only), each a
// sequential fmaf over its k; with more than one chunk the partial sums go to part[z][M][N] and
// gemm_chunk_reduce_kernel adds them in chunk order.  Tile loads are coalesced along whichever
// index of an operand has unit stride.
constexpr int GBM = 64, GBN = 64, GBK = 16;
constexpr int kGemmThreads = 256;
constexpr int kGemmTargetCTAs = 304;  // two 64 x 64 tiles per SM of a 152-SM GPU

struct GemmTileRegs {
    float v[GBM * GBK / kGemmThreads];
};

// Thread's share of the K tile [k0, k0 + GBK) of rows [row0, row0 + GBM): element e = tid + 256 q.
__device__ __forceinline__ void gemm_fetch(const float* __restrict__ X, int64_t s_row, int64_t s_k, int row0, int rows,
                                           int k0, int kend, GemmTileRegs& t)
{
#pragma unroll
    for (int q = 0; q < GBM * GBK / kGemmThreads; ++q) {
        const int e = threadIdx.x + kGemmThreads * q;
        const int r = s_k == 1 ? e / GBK : e % GBM, k = s_k == 1 ? e % GBK : e / GBM;
        const int row = row0 + r, kk = k0 + k;
        t.v[q] = (row < rows && kk < kend) ? __ldg(X + (int64_t)row * s_row + (int64_t)kk * s_k) : 0.f;
    }
}

__device__ __forceinline__ void gemm_stash(int64_t s_k, const GemmTileRegs& t, float (*dst)[GBM + 4])
{
#pragma unroll
    for (int q = 0; q < GBM * GBK / kGemmThreads; ++q) {
        const int e = threadIdx.x + kGemmThreads * q;
        const int r = s_k == 1 ? e / GBK : e % GBM, k = s_k == 1 ? e % GBK : e / GBM;
        dst[k][r] = t.v[q];
    }
}

__global__ void __launch_bounds__(kGemmThreads) gemm_f32_kernel(const float* __restrict__ A, int64_t sam, int64_t sak,
                                                                const float* __restrict__ B, int64_t sbn, int64_t sbk,
                                                                const float* __restrict__ bias, float* __restrict__ out,
                                                                int64_t ldo, int M, int N, int K, int kchunk,
                                                                float* __restrict__ part)
{
    __shared__ __align__(16) float As[2][GBK][GBM + 4], Bs[2][GBK][GBN + 4];
    const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;  // thread owns rows 4ty.., columns 4tx..
    const int m0 = blockIdx.y * GBM, n0 = blockIdx.x * GBN;
    const int kb = blockIdx.z * kchunk, ke = min(K, kb + kchunk);
    float acc[4][4] = {};
    GemmTileRegs ra, rb;
    gemm_fetch(A, sam, sak, m0, M, kb, ke, ra);
    gemm_fetch(B, sbn, sbk, n0, N, kb, ke, rb);
    int buf = 0;
    for (int k0 = kb; k0 < ke; k0 += GBK, buf ^= 1) {
        gemm_stash(sak, ra, As[buf]);
        gemm_stash(sbk, rb, Bs[buf]);
        __syncthreads();
        if (k0 + GBK < ke) {  // next tile in flight during the multiply
            gemm_fetch(A, sam, sak, m0, M, k0 + GBK, ke, ra);
            gemm_fetch(B, sbn, sbk, n0, N, k0 + GBK, ke, rb);
        }
#pragma unroll
        for (int k = 0; k < GBK; ++k) {
            const float4 a = *reinterpret_cast<const float4*>(&As[buf][k][4 * ty]);
            const float4 b = *reinterpret_cast<const float4*>(&Bs[buf][k][4 * tx]);
            const float av[4] = {a.x, a.y, a.z, a.w}, bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
        }
    }
    float* dst = part ? part + (int64_t)blockIdx.z * M * N : out;
    const int64_t ld = part ? N : ldo;
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int m = m0 + 4 * ty + i, n = n0 + 4 * tx + j;
            if (m < M && n < N) dst[(int64_t)m * ld + n] = part ? acc[i][j] : acc[i][j] + (bias ? bias[n] : 0.f);
        }
}

// out[m, n] = sum over chunks z = 0..nz-1 in order of part[z][m][n] (+ bias[n]).
__global__ void __launch_bounds__(256) gemm_chunk_reduce_kernel(const float* __restrict__ part, int nz, int M, int N,
                                                                const float* __restrict__ bias, float* __restrict__ out,
                                                                int64_t ldo)
{
    const int64_t total = (int64_t)M * N;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        float v = part[i];
        for (int z = 1; z < nz; ++z) v += part[z * total + i];
        const int m = (int)(i / N), n = (int)(i % N);
        out[(int64_t)m * ldo + n] = v + (bias ? bias[n] : 0.f);
    }
}

// K-chunking of an M x N x K head GEMM: enough chunks for ~kGemmTargetCTAs CTAs, at least
// four K tiles per chunk.  Returns the chunk length; *nz receives the chunk count.
int gemm_chunking(int M, int N, int K, int* nz)
{
    const int tiles = ((M + GBM - 1) / GBM) * ((N + GBN - 1) / GBN);
    int z = (kGemmTargetCTAs + tiles - 1) / tiles;
    const int zmax = std::max(1, (K + 4 * GBK - 1) / (4 * GBK));
    z = std::min(std::max(z, 1), zmax);
    int kchunk = (K + z - 1) / z;
    kchunk = (kchunk + GBK - 1) / GBK * GBK;
    *nz = (K + kchunk - 1) / kchunk;
    return kchunk;
}

size_t gemm_part_floats(int M, int N, int K)
{
    int nz;
    gemm_chunking(M, N, K, &nz);
    return nz > 1 ? (size_t)nz * M * N : 0;
}

int gemm_f32(const float* A, int64_t sam, int64_t sak, const float* B, int64_t sbn, int64_t sbk, const float* bias,
             float* out, int64_t ldo, int M, int N, int K, float* part, cudaStream_t s, const char* what)
{
    int nz;
    const int kchunk = gemm_chunking(M, N, K, &nz);
    dim3 g((N + GBN - 1) / GBN, (M + GBM - 1) / GBM, nz);
    gemm_f32_kernel<<<g, kGemmThreads, 0, s>>>(A, sam, sak, B, sbn, sbk, bias, out, ldo, M, N, K, kchunk,
                                                nz > 1 ? part : nullptr);
    int rc = dbl::launch_check(what);
    if (rc || nz == 1) return rc;
    const int64_t total = (int64_t)M * N;
    const int blocks = (int)std::min<int64_t>((total + 255) / 256, (int64_t)dbl::sm_count() * 8);
    gemm_chunk_reduce_kernel<<<blocks, 256, 0, s>>>(part, nz, M, N, bias, out, ldo);
    return dbl::launch_check(what);
}

// One warp per row: loss_n = logsumexp(l) - l[label]; dl = (softmax - onehot) * S/n (in place), S the
// loss scale (1 without loss scaling).
__global__ void softmax_ce_kernel(float* __restrict__ logits, const int32_t* __restrict__ labels, int n, int J,
                                  float* __restrict__ row_loss, const float* __restrict__ loss_scale)
{
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) / 32, lane = threadIdx.x % 32;
    if (warp >= n) return;
    float* l = logits + (int64_t)warp * J;
    float mx = -FLT_MAX;
    for (int j = lane; j < J; j += 32) mx = fmaxf(mx, l[j]);
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float z = 0.f;
    for (int j = lane; j < J; j += 32) z += expf(l[j] - mx);
    for (int o = 16; o; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    const float lse = mx + logf(z);
    const int lab = labels[warp];
    if (lane == 0) row_loss[warp] = lse - l[lab];
    const float invn = (loss_scale ? *loss_scale : 1.0f) / (float)n;
    for (int j = lane; j < J; j += 32) l[j] = (expf(l[j] - lse) - (j == lab ? 1.f : 0.f)) * invn;
}

// loss = mean(row_loss) (block 0, fixed order); db[j] = sum_n dl[n, j] (blocks 1..: 32 columns each,
// warp w adding rows w, w + 8, ... in order, then the eight warp sums added in warp order).  Each
// column's rows are spread over eight warps instead of one thread's chain of n dependent adds.
constexpr int kHeadRedCols = 32;
__global__ void __launch_bounds__(256) head_reduce_kernel(const float* __restrict__ row_loss, const float* __restrict__ dl,
                                                          int n, int J, float* __restrict__ loss, float* __restrict__ db)
{
    __shared__ float red[256];
    if (blockIdx.x == 0) {
        float s = 0.f;
        for (int i = threadIdx.x; i < n; i += blockDim.x) s += row_loss[i];
        red[threadIdx.x] = s;
        __syncthreads();
        for (int w = blockDim.x / 2; w; w >>= 1) {
            if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
            __syncthreads();
        }
        if (threadIdx.x == 0) *loss = red[0] / (float)n;
        return;
    }
    const int lane = threadIdx.x % 32, w = threadIdx.x / 32;
    const int j = (blockIdx.x - 1) * kHeadRedCols + lane;
    float s = 0.f;
    if (j < J)
        for (int i = w; i < n; i += 8) s += dl[(int64_t)i * J + j];
    red[threadIdx.x] = s;
    __syncthreads();
    if (w == 0 && j < J) {
        float t = red[lane];
#pragma unroll
        for (int k = 1; k < 8; ++k) t += red[k * 32 + lane];
        db[j] = t;
    }
}

// The same two passes with one CTA per image, blockDim = S slices x (C/8) channel groups: thread
// (slice s, group g) takes the rows i = s, s + S, ... of its image (consecutive threads on
// consecutive 16-byte vectors of a row).  Forward: each slice adds its rows in order, then the S
// slice sums are added in slice order.  Backward: each thread computes its 8 gradients once and
// writes them to its rows.  (One thread per (image, group) walking all hw rows, or loading its
// 16 fp32 factors again for every row, left these passes at a fifth of HBM.)
__device__ __forceinline__ int pool_slices(int groups) { return groups >= 1024 ? 1 : min(8, 1024 / groups); }

__global__ void __launch_bounds__(1024) avgpool_img_kernel(const act_t* __restrict__ x, float* __restrict__ feat,
                                                           int hw, int C, Dropout dp)
{
    extern __shared__ float slice_sum[];  // [S][C]
    const int groups = C / 8, S = pool_slices(groups);
    const int g = threadIdx.x % groups, sl = threadIdx.x / groups;
    const int b = blockIdx.x;
    float acc[8] = {};
    for (int i = sl; i < hw; i += S) {
        float f[8];
        unpack8(__ldg(reinterpret_cast<const uint4*>(x + ((int64_t)b * hw + i) * C) + g), f);
#pragma unroll
        for (int k = 0; k < 8; ++k) acc[k] += f[k];
    }
#pragma unroll
    for (int k = 0; k < 8; ++k) slice_sum[sl * C + 8 * g + k] = acc[k];
    __syncthreads();
    if (sl != 0) return;
    for (int q = 1; q < S; ++q)
#pragma unroll
        for (int k = 0; k < 8; ++k) acc[k] += slice_sum[q * C + 8 * g + k];
    const float inv = 1.0f / (float)hw;
    if (dp.thr) {
        const uint64_t st = *dp.step;
        const uint64_t q = (uint64_t)b * (uint64_t)(C / 4) + 2 * (uint64_t)g;
        const unsigned bits = dropout_keep4(dp.seed, st, q, dp.thr) | dropout_keep4(dp.seed, st, q + 1, dp.thr) << 4;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const float m = (bits >> k) & 1 ? dp.scale : 0.f;
            dp.mult[(int64_t)b * C + 8 * g + k] = m;
            feat[(int64_t)b * C + 8 * g + k] = acc[k] * inv * m;
        }
    } else {
#pragma unroll
        for (int k = 0; k < 8; ++k) feat[(int64_t)b * C + 8 * g + k] = acc[k] * inv;
    }
}

// step (or nullptr): the dropout step counter, advanced once here so that the next call draws a
// fresh mask (every read of it in this call has happened in the forward pool)
__global__ void __launch_bounds__(1024) avgpool_bwd_img_kernel(const float* __restrict__ df, act_t* __restrict__ dx,
                                                               int hw, int C, const float* __restrict__ mult,
                                                               uint64_t* __restrict__ step)
{
    if (step && blockIdx.x == 0 && threadIdx.x == 0) *step += 1;
    const int groups = C / 8, S = pool_slices(groups);
    const int g = threadIdx.x % groups, sl = threadIdx.x / groups;
    const int b = blockIdx.x;
    const float inv = 1.0f / (float)hw;
    float f[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const int64_t e = (int64_t)b * C + 8 * g + k;
        f[k] = (mult ? df[e] * mult[e] : df[e]) * inv;
    }
    const uint4 v = pack8(f);
    uint4* row = reinterpret_cast<uint4*>(dx + (int64_t)b * hw * C) + g;
    for (int i = sl; i < hw; i += S) row[(int64_t)i * groups] = v;
}

// dx[n, i, c] = df[n, c] / hw, with dropout (df[n, c] * mult[n, c]) / hw
__global__ void __launch_bounds__(256) avgpool_bwd_kernel(const float* __restrict__ df, act_t* __restrict__ dx,
                                                          int n, int hw, int C, const float* __restrict__ mult,
                                                          uint64_t* __restrict__ step)
{
    if (step && blockIdx.x == 0 && threadIdx.x == 0) *step += 1;  // as in avgpool_bwd_img_kernel
    const int groups = C / 8;
    const int64_t total = (int64_t)n * hw * groups;
    const float inv = 1.0f / (float)hw;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int g = (int)(t % groups);
        const int b = (int)(t / groups / hw);
        float f[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int64_t e = (int64_t)b * C + 8 * g + k;
            f[k] = (mult ? df[e] * mult[e] : df[e]) * inv;
        }
        reinterpret_cast<uint4*>(dx)[t] = pack8(f);
    }
}

}  // namespace

extern "C" {

int dbl_maxpool_fwd(int32_t n, int32_t h, int32_t w, int32_t c, const void* x, void* y, uint8_t* argmax, void* stream)
{
    using namespace dbl;
    if (n < 0 || h <= 0 || w <= 0 || c <= 0 || !x || !y || !argmax)
        return set_error(DBL_ERR_INVALID, "maxpool_fwd: bad arguments");
    if (c % 8) return set_error(DBL_ERR_INVALID, "maxpool_fwd: channels must be a multiple of 8");
    if (!aligned16(x) || !aligned16(y) || (reinterpret_cast<uintptr_t>(argmax) & 7))
        return set_error(DBL_ERR_INVALID, "maxpool_fwd: misaligned pointer");
    const int P = (h + 2 - 3) / 2 + 1, Q = (w + 2 - 3) / 2 + 1;
    if ((int64_t)n * h * w * (c / 8) >= (int64_t)1 << 31)
        return set_error(DBL_ERR_UNSUPPORTED, "maxpool_fwd: tensor too large for 32-bit indexing");
    if (n == 0) return DBL_OK;
    maxpool_fwd_kernel<<<grid_for((int64_t)n * P * Q * (c / 8), 256), 256, 0, as_stream(stream)>>>(
        static_cast<const act_t*>(x), static_cast<act_t*>(y), argmax, n, h, w, c, P, Q);
    return launch_check("maxpool_fwd launch");
}

int dbl_bn_relu_maxpool_fwd(const dbl_bn_shape* s, int32_t n, int32_t h, int32_t w, const void* x,
                            const float* ch_sum, const float* ch_sumsq, const float* gamma, const float* beta,
                            float* save_mean, float* save_invstd, void* y, uint8_t* argmax, void* stream)
{
    using namespace dbl;
    if (!s || n <= 0 || h <= 0 || w <= 0 || !x || !y || !argmax || !ch_sum || !ch_sumsq || !gamma || !beta ||
        !save_mean || !save_invstd)
        return set_error(DBL_ERR_INVALID, "bn_relu_maxpool_fwd: bad arguments");
    const int c = s->c;
    if (c <= 0 || c % 8 || !s->relu || s->count != (int64_t)n * h * w)
        return set_error(DBL_ERR_INVALID, "bn_relu_maxpool_fwd: shape must be [n*h*w, c], c a multiple of 8, relu set");
    if (c > 8192) return set_error(DBL_ERR_UNSUPPORTED, "bn_relu_maxpool_fwd: at most 8192 channels");
    if (!aligned16(x) || !aligned16(y) || (reinterpret_cast<uintptr_t>(argmax) & 7))
        return set_error(DBL_ERR_INVALID, "bn_relu_maxpool_fwd: misaligned pointer");
    const int P = (h + 2 - 3) / 2 + 1, Q = (w + 2 - 3) / 2 + 1;
    if ((int64_t)n * h * w * (c / 8) >= (int64_t)1 << 31)
        return set_error(DBL_ERR_UNSUPPORTED, "bn_relu_maxpool_fwd: tensor too large for 32-bit indexing");
    cudaStream_t st = as_stream(stream);
    int rc = bn_fwd_finalize(s->count, c, s->eps, ch_sum, ch_sumsq, save_mean, save_invstd, st);
    if (rc) return rc;
    // a block size that is a multiple of the channel groups: each thread keeps its group
    const int groups = c / 8, block = groups * std::max(1, 256 / groups);
    bn_relu_maxpool_fwd_kernel<<<grid_for((int64_t)n * P * Q, block / groups), block, 0, st>>>(
        static_cast<const act_t*>(x), gamma, beta, save_mean, save_invstd, static_cast<act_t*>(y),
        argmax, n, h, w, c, P, Q);
    return launch_check("bn_relu_maxpool_fwd launch");
}

int dbl_maxpool_bwd(int32_t n, int32_t h, int32_t w, int32_t c, const void* dy, const void* dy2,
                    const uint8_t* argmax, void* dx, void* stream)
{
    using namespace dbl;
    if (n < 0 || h <= 0 || w <= 0 || c <= 0 || !dy || !dx || !argmax)
        return set_error(DBL_ERR_INVALID, "maxpool_bwd: bad arguments");
    if (c % 8) return set_error(DBL_ERR_INVALID, "maxpool_bwd: channels must be a multiple of 8");
    if (!aligned16(dy) || !aligned16(dx) || (dy2 && !aligned16(dy2)) || (reinterpret_cast<uintptr_t>(argmax) & 7))
        return set_error(DBL_ERR_INVALID, "maxpool_bwd: misaligned pointer");
    const int P = (h + 2 - 3) / 2 + 1, Q = (w + 2 - 3) / 2 + 1;
    if ((int64_t)n * h * w * (c / 8) >= (int64_t)1 << 31)
        return set_error(DBL_ERR_UNSUPPORTED, "maxpool_bwd: tensor too large for 32-bit indexing");
    if (n == 0) return DBL_OK;
    if (c > 8192) return set_error(DBL_ERR_UNSUPPORTED, "maxpool_bwd: at most 8192 channels");
    // a block size that is a multiple of the channel groups: each thread keeps its group
    const int groups = c / 8, block = groups * std::max(1, 256 / groups);
    maxpool_bwd_kernel<<<grid_for((int64_t)n * ((h + 1) / 2) * ((w + 1) / 2), block / groups), block, 0,
                         as_stream(stream)>>>(
        static_cast<const act_t*>(dy), static_cast<const act_t*>(dy2), argmax,
        static_cast<act_t*>(dx), n, h, w, c, P, Q);
    return launch_check("maxpool_bwd launch");
}

size_t dbl_head_workspace_bytes(int32_t n, int32_t c, int32_t classes)
{
    if (n <= 0 || c <= 0 || classes <= 0) return 0;
    // feat [n,c], logits/dlogits [n,classes], df [n,c], row_loss [n], dropout multipliers [n,c],
    // then the K-chunk partial sums of the largest of the three GEMMs
    const size_t f = (size_t)n * c * 3 + (size_t)n * classes + (size_t)n;
    const size_t part = std::max({gemm_part_floats(n, classes, c), gemm_part_floats(classes, c, n),
                                  gemm_part_floats(n, c, classes)});
    return (((f + 3) / 4 * 4 + part) * sizeof(float) + 255) / 256 * 256;
}

}  // extern "C"

namespace {

int head_fwd_bwd(int32_t n, int32_t hw, int32_t c, int32_t classes, const void* x, const float* fc_w, const float* fc_b,
                 const int32_t* labels, float drop_rate, uint64_t seed, uint64_t* step, const float* loss_scale,
                 float* loss, float* dfc_w, float* dfc_b, void* dx, void* ws, size_t ws_bytes, void* stream,
                 const char* name)
{
    using namespace dbl;
    if (n <= 0 || hw <= 0 || c <= 0 || classes <= 0 || !x || !fc_w || !fc_b || !labels || !loss || !dfc_w || !dfc_b ||
        !dx)
        return set_error(DBL_ERR_INVALID, "%s: bad arguments", name);
    if (c % 8 || !aligned16(x) || !aligned16(dx))
        return set_error(DBL_ERR_INVALID, "%s: channels must be a multiple of 8, tensors 16-byte aligned", name);
    if (!(drop_rate >= 0.f && drop_rate < 1.f))
        return set_error(DBL_ERR_INVALID, "%s: dropout rate %g outside [0, 1)", name, (double)drop_rate);
    if (drop_rate > 0.f && (!step || (reinterpret_cast<uintptr_t>(step) & 7)))
        return set_error(DBL_ERR_INVALID, "%s: dropout needs an 8-byte aligned device step counter", name);
    const size_t need = dbl_head_workspace_bytes(n, c, classes);
    if (!ws || ws_bytes < need) return set_error(DBL_ERR_WORKSPACE, "%s: workspace %zu < %zu", name, ws_bytes, need);
    float* feat = static_cast<float*>(ws);
    float* logits = feat + (size_t)n * c;
    float* df = logits + (size_t)n * classes;
    float* row_loss = df + (size_t)n * c;
    float* mult = row_loss + (size_t)n;
    float* part = feat + ((size_t)n * c * 3 + (size_t)n * classes + (size_t)n + 3) / 4 * 4;
    Dropout dp{0u, 1.f, seed, step, mult};
    if (drop_rate > 0.f) {
        dp.thr = (uint32_t)floor((double)drop_rate * 4294967296.0);
        dp.scale = (float)(1.0 / (1.0 - (double)drop_rate));
    }
    cudaStream_t s = as_stream(stream);
    int rc;
    const int groups = c / 8;
    const bool per_image = groups <= 1024;  // one CTA per image (at most 1024 threads)
    const int S = groups >= 1024 ? 1 : std::min(8, 1024 / groups);
    if (per_image)
        avgpool_img_kernel<<<n, S * groups, (size_t)S * c * sizeof(float), s>>>(static_cast<const act_t*>(x), feat,
                                                                                 hw, c, dp);
    else
        avgpool_kernel<<<grid_for((int64_t)n * groups, 256), 256, 0, s>>>(static_cast<const act_t*>(x), feat, n, hw,
                                                                           c, dp);
    if ((rc = launch_check("avgpool launch"))) return rc;
    // logits = feat * W^T + b
    if ((rc = gemm_f32(feat, c, 1, fc_w, c, 1, fc_b, logits, classes, n, classes, c, part, s, "fc fwd launch")))
        return rc;
    softmax_ce_kernel<<<(n * 32 + 255) / 256, 256, 0, s>>>(logits, labels, n, classes, row_loss, loss_scale);
    if ((rc = launch_check("softmax_ce launch"))) return rc;
    head_reduce_kernel<<<1 + (classes + kHeadRedCols - 1) / kHeadRedCols, 256, 0, s>>>(row_loss, logits, n, classes,
                                                                                        loss, dfc_b);
    if ((rc = launch_check("head reduce launch"))) return rc;
    // dW[j, c] = sum_n dl[n, j] feat[n, c]
    if ((rc = gemm_f32(logits, 1, classes, feat, 1, c, nullptr, dfc_w, c, classes, c, n, part, s, "fc dW launch")))
        return rc;
    // df[n, c] = sum_j dl[n, j] W[j, c]
    if ((rc = gemm_f32(logits, classes, 1, fc_w, 1, c, nullptr, df, c, n, c, classes, part, s, "fc dX launch")))
        return rc;
    // with dropout, the pool's backward also advances the step counter (the next call draws a fresh mask)
    uint64_t* adv = dp.thr ? step : nullptr;
    if (per_image)
        avgpool_bwd_img_kernel<<<n, S * groups, 0, s>>>(df, static_cast<act_t*>(dx), hw, c, dp.thr ? mult : nullptr,
                                                        adv);
    else
        avgpool_bwd_kernel<<<grid_for((int64_t)n * hw * groups, 256), 256, 0, s>>>(df, static_cast<act_t*>(dx), n, hw,
                                                                                    c, dp.thr ? mult : nullptr, adv);
    return launch_check("avgpool_bwd launch");
}

}  // namespace

extern "C" {

int dbl_head_fwd_bwd(int32_t n, int32_t hw, int32_t c, int32_t classes, const void* x, const float* fc_w,
                     const float* fc_b, const int32_t* labels, float* loss, float* dfc_w, float* dfc_b, void* dx,
                     void* ws, size_t ws_bytes, void* stream)
{
    return head_fwd_bwd(n, hw, c, classes, x, fc_w, fc_b, labels, 0.f, 0, nullptr, nullptr, loss, dfc_w, dfc_b, dx, ws,
                        ws_bytes, stream, "head_fwd_bwd");
}

int dbl_head_fwd_bwd_ex(int32_t n, int32_t hw, int32_t c, int32_t classes, const void* x, const float* fc_w,
                        const float* fc_b, const int32_t* labels, const dbl_head_opts* opts, float* loss, float* dfc_w,
                        float* dfc_b, void* dx, void* ws, size_t ws_bytes, void* stream)
{
    if (!opts) return dbl::set_error(DBL_ERR_INVALID, "head_fwd_bwd_ex: null options");
    return head_fwd_bwd(n, hw, c, classes, x, fc_w, fc_b, labels, opts->drop_rate, opts->seed, opts->step,
                        opts->loss_scale, loss, dfc_w, dfc_b, dx, ws, ws_bytes, stream, "head_fwd_bwd_ex");
}

int dbl_dropout_mask(int32_t n, int32_t c, float drop_rate, uint64_t seed, const uint64_t* step, uint8_t* keep,
                     void* stream)
{
    using namespace dbl;
    if (n < 0 || c <= 0 || c % 4 || !keep || (reinterpret_cast<uintptr_t>(keep) & 3))
        return set_error(DBL_ERR_INVALID, "dropout_mask: bad arguments (c a multiple of 4, keep 4-byte aligned)");
    if (!(drop_rate >= 0.f && drop_rate < 1.f))
        return set_error(DBL_ERR_INVALID, "dropout_mask: rate %g outside [0, 1)", (double)drop_rate);
    const uint32_t thr = drop_rate > 0.f ? (uint32_t)floor((double)drop_rate * 4294967296.0) : 0u;
    if (thr && (!step || (reinterpret_cast<uintptr_t>(step) & 7)))
        return set_error(DBL_ERR_INVALID, "dropout_mask: needs an 8-byte aligned device step counter");
    if (n == 0) return DBL_OK;
    dropout_mask_kernel<<<grid_for((int64_t)n * (c / 4), 256), 256, 0, as_stream(stream)>>>(n, c, thr, seed, step, keep);
    return launch_check("dropout_mask launch");
}

}  // extern "C"
