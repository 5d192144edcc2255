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
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 t = __bfloat1622float2(h[k]);
        f[2 * k] = t.x;
        f[2 * k + 1] = t.y;
    }
}

__device__ __forceinline__ uint4 pack8(const float (&f)[8])
{
    uint4 v;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&v);
#pragma unroll
    for (int k = 0; k < 4; ++k) h[k] = __floats2bfloat162_rn(f[2 * k], f[2 * k + 1]);
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
__global__ void __launch_bounds__(256) maxpool_fwd_kernel(const __nv_bfloat16* __restrict__ x,
                                                          __nv_bfloat16* __restrict__ y, uint8_t* __restrict__ arg,
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
__global__ void __launch_bounds__(256)
    bn_relu_maxpool_fwd_kernel(const __nv_bfloat16* __restrict__ x, const float* __restrict__ gamma,
                               const float* __restrict__ beta, const float* __restrict__ mean,
                               const float* __restrict__ invstd, __nv_bfloat16* __restrict__ y,
                               uint8_t* __restrict__ arg, int n, int H, int W, int C, int P, int Q)
{
    const unsigned groups = (unsigned)C / 8u;
    const unsigned total = (unsigned)n * P * Q * groups;
    // a thread keeps its channel group across the grid-stride loop when the stride is a multiple of groups
    for (unsigned t = blockIdx.x * blockDim.x + threadIdx.x; t < total; t += gridDim.x * blockDim.x) {
        const unsigned g = t % groups;
        unsigned pix = t / groups;
        const int q = (int)(pix % (unsigned)Q);
        pix /= (unsigned)Q;
        const int p = (int)(pix % (unsigned)P);
        const int b = (int)(pix / (unsigned)P);
        float sc[8], sh[8];
#pragma unroll
        for (int k = 0; k < 8; ++k)
            dbl::dev::bn_scale_shift(gamma[8 * g + k], beta[8 * g + k], mean[8 * g + k], invstd[8 * g + k], sc[k],
                                     sh[k]);
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
                for (int k = 0; k < 8; ++k) {
                    const float o = __fadd_rn(__fmaf_rn(f[k], sc[k], sh[k]), 0.f);
                    const float a = __bfloat162float(__float2bfloat16_rn(o > 0.f ? o : 0.f));
                    if (a > best[k]) {  // strict: the first maximum in (r, s) order wins ties
                        best[k] = a;
                        bi[k] = (uint8_t)(r * 3 + s);
                    }
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

// Gather form over 2x2 blocks of input pixels: block (i, j) = rows 2i..2i+1,
// cols 2j..2j+1 is covered by windows (i..i+1, j..j+1); window (p, q) reaches
// input (h, w) at tap (h - 2p + 1, w - 2q + 1).  Each window's argmax and
// gradient are read once per block, and every input pixel sums its windows in
// (p, q) order.
__global__ void __launch_bounds__(256)
    maxpool_bwd_kernel(const __nv_bfloat16* __restrict__ dy, const __nv_bfloat16* __restrict__ dy2,
                       const uint8_t* __restrict__ arg, __nv_bfloat16* __restrict__ dx, int n, int H, int W, int C,
                       int P, int Q)
{
    const unsigned groups = (unsigned)C / 8u;
    const int BH = (H + 1) / 2, BW = (W + 1) / 2;
    const unsigned total = (unsigned)n * BH * BW * groups;
    for (unsigned t = blockIdx.x * blockDim.x + threadIdx.x; t < total; t += gridDim.x * blockDim.x) {
        const unsigned g = t % groups;
        unsigned pix = t / groups;
        const int j = (int)(pix % (unsigned)BW);
        pix /= (unsigned)BW;
        const int i = (int)(pix % (unsigned)BH);
        const int b = (int)(pix / (unsigned)BH);
        float acc[4][8] = {};
        for (int dp = 0; dp < 2; ++dp) {
            const int p = i + dp;
            if (p >= P) continue;
            for (int dq = 0; dq < 2; ++dq) {
                const int q = j + dq;
                if (q >= Q) continue;
                const int64_t o = (((int64_t)b * P + p) * Q + q) * C + 8 * g;
                const uint2 a = __ldg(reinterpret_cast<const uint2*>(arg + o));
                const uint8_t* ab = reinterpret_cast<const uint8_t*>(&a);
                float f[8];
                unpack8(__ldg(reinterpret_cast<const uint4*>(dy + o)), f);
                if (dy2) {
                    float f2[8];
                    unpack8(__ldg(reinterpret_cast<const uint4*>(dy2 + o)), f2);
#pragma unroll
                    for (int k = 0; k < 8; ++k) f[k] += f2[k];
                }
#pragma unroll
                for (int dh = 0; dh < 2; ++dh) {
                    const int r = 2 * i + dh - 2 * p + 1;  // tap row of input row 2i+dh in window row p
                    if (r < 0 || r > 2) continue;
#pragma unroll
                    for (int dw = 0; dw < 2; ++dw) {
                        const int sx = 2 * j + dw - 2 * q + 1;
                        if (sx < 0 || sx > 2) continue;
                        const uint8_t me = (uint8_t)(r * 3 + sx);
#pragma unroll
                        for (int k = 0; k < 8; ++k)
                            if (ab[k] == me) acc[dh * 2 + dw][k] += f[k];
                    }
                }
            }
        }
#pragma unroll
        for (int dh = 0; dh < 2; ++dh) {
            const int h = 2 * i + dh;
            if (h >= H) continue;
#pragma unroll
            for (int dw = 0; dw < 2; ++dw) {
                const int w = 2 * j + dw;
                if (w >= W) continue;
                *reinterpret_cast<uint4*>(dx + (((int64_t)b * H + h) * W + w) * C + 8 * g) = pack8(acc[dh * 2 + dw]);
            }
        }
    }
}

// ----------------------------------------------------------------------------- head
// feat[n, c] = mean over hw of x[n, hw, c]
__global__ void __launch_bounds__(256) avgpool_kernel(const __nv_bfloat16* __restrict__ x, float* __restrict__ feat,
                                                      int n, int hw, int C)
{
    const int groups = C / 8;
    const int64_t total = (int64_t)n * groups;
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
#pragma unroll
        for (int k = 0; k < 8; ++k) feat[(int64_t)b * C + 8 * g + k] = acc[k] * inv;
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

// One warp per row: loss_n = logsumexp(l) - l[label]; dl = (softmax - onehot)/n (in place).
__global__ void softmax_ce_kernel(float* __restrict__ logits, const int32_t* __restrict__ labels, int n, int J,
                                  float* __restrict__ row_loss)
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
    const float invn = 1.0f / (float)n;
    for (int j = lane; j < J; j += 32) l[j] = (expf(l[j] - lse) - (j == lab ? 1.f : 0.f)) * invn;
}

// loss = mean(row_loss) (one block, fixed order); db[j] = sum_n dl[n, j].
__global__ void head_reduce_kernel(const float* __restrict__ row_loss, const float* __restrict__ dl, int n, int J,
                                   float* __restrict__ loss, float* __restrict__ db)
{
    if (blockIdx.x == 0) {
        __shared__ float red[256];
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
    const int j = (blockIdx.x - 1) * blockDim.x + threadIdx.x;
    if (j >= J) return;
    float s = 0.f;
    for (int i = 0; i < n; ++i) s += dl[(int64_t)i * J + j];
    db[j] = s;
}

// dx[n, i, c] = df[n, c] / hw
__global__ void __launch_bounds__(256) avgpool_bwd_kernel(const float* __restrict__ df, __nv_bfloat16* __restrict__ dx,
                                                          int n, int hw, int C)
{
    const int groups = C / 8;
    const int64_t total = (int64_t)n * hw * groups;
    const float inv = 1.0f / (float)hw;
    for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (int64_t)gridDim.x * blockDim.x) {
        const int g = (int)(t % groups);
        const int b = (int)(t / groups / hw);
        float f[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) f[k] = df[(int64_t)b * C + 8 * g + k] * inv;
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
        static_cast<const __nv_bfloat16*>(x), static_cast<__nv_bfloat16*>(y), argmax, n, h, w, c, P, Q);
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
    if (!aligned16(x) || !aligned16(y) || (reinterpret_cast<uintptr_t>(argmax) & 7))
        return set_error(DBL_ERR_INVALID, "bn_relu_maxpool_fwd: misaligned pointer");
    const int P = (h + 2 - 3) / 2 + 1, Q = (w + 2 - 3) / 2 + 1;
    if ((int64_t)n * h * w * (c / 8) >= (int64_t)1 << 31)
        return set_error(DBL_ERR_UNSUPPORTED, "bn_relu_maxpool_fwd: tensor too large for 32-bit indexing");
    cudaStream_t st = as_stream(stream);
    int rc = bn_fwd_finalize(s->count, c, s->eps, ch_sum, ch_sumsq, save_mean, save_invstd, st);
    if (rc) return rc;
    bn_relu_maxpool_fwd_kernel<<<grid_for((int64_t)n * P * Q * (c / 8), 256), 256, 0, st>>>(
        static_cast<const __nv_bfloat16*>(x), gamma, beta, save_mean, save_invstd, static_cast<__nv_bfloat16*>(y),
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
    maxpool_bwd_kernel<<<grid_for((int64_t)n * ((h + 1) / 2) * ((w + 1) / 2) * (c / 8), 256), 256, 0,
                         as_stream(stream)>>>(
        static_cast<const __nv_bfloat16*>(dy), static_cast<const __nv_bfloat16*>(dy2), argmax,
        static_cast<__nv_bfloat16*>(dx), n, h, w, c, P, Q);
    return launch_check("maxpool_bwd launch");
}

size_t dbl_head_workspace_bytes(int32_t n, int32_t c, int32_t classes)
{
    if (n <= 0 || c <= 0 || classes <= 0) return 0;
    // feat [n,c], logits/dlogits [n,classes], df [n,c], row_loss [n], then the K-chunk partial
    // sums of the largest of the three GEMMs
    const size_t f = (size_t)n * c * 2 + (size_t)n * classes + (size_t)n;
    const size_t part = std::max({gemm_part_floats(n, classes, c), gemm_part_floats(classes, c, n),
                                  gemm_part_floats(n, c, classes)});
    return (((f + 3) / 4 * 4 + part) * sizeof(float) + 255) / 256 * 256;
}

int dbl_head_fwd_bwd(int32_t n, int32_t hw, int32_t c, int32_t classes, const void* x, const float* fc_w,
                     const float* fc_b, const int32_t* labels, float* loss, float* dfc_w, float* dfc_b, void* dx,
                     void* ws, size_t ws_bytes, void* stream)
{
    using namespace dbl;
    if (n <= 0 || hw <= 0 || c <= 0 || classes <= 0 || !x || !fc_w || !fc_b || !labels || !loss || !dfc_w || !dfc_b ||
        !dx)
        return set_error(DBL_ERR_INVALID, "head_fwd_bwd: bad arguments");
    if (c % 8 || !aligned16(x) || !aligned16(dx))
        return set_error(DBL_ERR_INVALID, "head_fwd_bwd: channels must be a multiple of 8, tensors 16-byte aligned");
    const size_t need = dbl_head_workspace_bytes(n, c, classes);
    if (!ws || ws_bytes < need) return set_error(DBL_ERR_WORKSPACE, "head_fwd_bwd: workspace %zu < %zu", ws_bytes, need);
    float* feat = static_cast<float*>(ws);
    float* logits = feat + (size_t)n * c;
    float* df = logits + (size_t)n * classes;
    float* row_loss = df + (size_t)n * c;
    float* part = feat + ((size_t)n * c * 2 + (size_t)n * classes + (size_t)n + 3) / 4 * 4;
    cudaStream_t s = as_stream(stream);
    int rc;
    avgpool_kernel<<<grid_for((int64_t)n * (c / 8), 256), 256, 0, s>>>(static_cast<const __nv_bfloat16*>(x), feat, n,
                                                                       hw, c);
    if ((rc = launch_check("avgpool launch"))) return rc;
    // logits = feat * W^T + b
    if ((rc = gemm_f32(feat, c, 1, fc_w, c, 1, fc_b, logits, classes, n, classes, c, part, s, "fc fwd launch")))
        return rc;
    softmax_ce_kernel<<<(n * 32 + 255) / 256, 256, 0, s>>>(logits, labels, n, classes, row_loss);
    if ((rc = launch_check("softmax_ce launch"))) return rc;
    head_reduce_kernel<<<1 + (classes + 255) / 256, 256, 0, s>>>(row_loss, logits, n, classes, loss, dfc_b);
    if ((rc = launch_check("head reduce launch"))) return rc;
    // dW[j, c] = sum_n dl[n, j] feat[n, c]
    if ((rc = gemm_f32(logits, 1, classes, feat, 1, c, nullptr, dfc_w, c, classes, c, n, part, s, "fc dW launch")))
        return rc;
    // df[n, c] = sum_j dl[n, j] W[j, c]
    if ((rc = gemm_f32(logits, classes, 1, fc_w, 1, c, nullptr, df, c, n, c, classes, part, s, "fc dX launch")))
        return rc;
    avgpool_bwd_kernel<<<grid_for((int64_t)n * hw * (c / 8), 256), 256, 0, s>>>(df, static_cast<__nv_bfloat16*>(dx), n,
                                                                                hw, c);
    return launch_check("avgpool_bwd launch");
}

}  // extern "C"
