// resize.cu -- progressive resizing for the low-resolution sub-stages of
// cyclic progressive learning (Sec. 4.1): bilinear downsampling with
// half-pixel centres, fused with the cast to the network's input type and
// the zero channel padding (3 colour channels -> 8, one 16-byte pixel).
//
// Taps are integer-exact: output j of an axis reads source rows
// i0 = floor(num/den) and min(i0+1, in-1) with weight (num - i0*den)/den,
// num = (2j+1)*in - out, den = 2*out.  When in == out this is a plain copy.
#include "dbl_internal.cuh"

namespace {

struct Taps {
    int32_t i0, i1;
    float lam;
};

__device__ __forceinline__ Taps axis_taps(int32_t j, int32_t in, int32_t out)
{
    // 32-bit: the host limits sizes so that (2j+1)*in stays far below 2^31
    const int32_t num = (2 * j + 1) * in - out;
    const int32_t den = 2 * out;
    const int32_t a = num / den;
    Taps t;
    t.i0 = (int32_t)a;
    t.i1 = (int32_t)(a + 1 < in ? a + 1 : in - 1);
    t.lam = (float)(num - a * den) / (float)den;
    return t;
}

template <typename Tin>
__device__ __forceinline__ float ld_in(const Tin* p);
template <>
__device__ __forceinline__ float ld_in<float>(const float* p)
{
    return __ldg(p);
}
template <>
__device__ __forceinline__ float ld_in<act_t>(const act_t* p)
{
    return dbl::act::to_f(*p);
}

// One thread per output pixel; channels 0..c-1 interpolated, c..cs-1 zeroed.
template <typename Tin, typename Tout, int CMAX>
__global__ void __launch_bounds__(256) resize_kernel(const Tin* __restrict__ in, Tout* __restrict__ out, int32_t n,
                                                     int32_t hi, int32_t wi, int32_t c, int32_t ho, int32_t wo,
                                                     int32_t cs)
{
    // 32-bit index math: the host checks that n*ho*wo fits
    const unsigned total = (unsigned)n * ho * wo;
    for (unsigned pix = blockIdx.x * blockDim.x + threadIdx.x; pix < total; pix += gridDim.x * blockDim.x) {
        const int32_t x = (int32_t)(pix % (unsigned)wo);
        const unsigned t = pix / (unsigned)wo;
        const int32_t y = (int32_t)(t % (unsigned)ho);
        const int32_t b = (int32_t)(t / (unsigned)ho);
        const Taps ty = axis_taps(y, hi, ho), tx = axis_taps(x, wi, wo);
        const Tin* base = in + (int64_t)b * hi * wi * c;
        const Tin* pa = base + ((int64_t)ty.i0 * wi + tx.i0) * c;
        const Tin* pb = base + ((int64_t)ty.i0 * wi + tx.i1) * c;
        const Tin* pc = base + ((int64_t)ty.i1 * wi + tx.i0) * c;
        const Tin* pd = base + ((int64_t)ty.i1 * wi + tx.i1) * c;
        float v[CMAX];
#pragma unroll
        for (int ch = 0; ch < CMAX; ++ch) {
            v[ch] = 0.f;
            if (ch < c) {
                const float top = (1.f - tx.lam) * ld_in(pa + ch) + tx.lam * ld_in(pb + ch);
                const float bot = (1.f - tx.lam) * ld_in(pc + ch) + tx.lam * ld_in(pd + ch);
                v[ch] = (1.f - ty.lam) * top + ty.lam * bot;
            }
        }
        Tout* o = out + (int64_t)pix * cs;
        if constexpr (sizeof(Tout) == 2 && CMAX == 8) {
            if (cs == 8) {  // one 16-byte store per pixel
                act2_t q[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) q[k] = dbl::act::pack2(v[2 * k], v[2 * k + 1]);
                *reinterpret_cast<uint4*>(o) = *reinterpret_cast<uint4*>(q);
                continue;
            }
        }
        for (int ch = 0; ch < cs; ++ch) {
            const float val = ch < CMAX ? v[ch < CMAX ? ch : 0] : 0.f;
            if constexpr (sizeof(Tout) == 2)
                o[ch] = dbl::act::from_f(val);
            else
                o[ch] = val;
        }
    }
}

template <typename Tin, typename Tout>
int launch_resize(const void* in, void* out, int32_t n, int32_t hi, int32_t wi, int32_t c, int32_t ho, int32_t wo,
                  int32_t cs, cudaStream_t s)
{
    const int64_t total = (int64_t)n * ho * wo;
    const int threads = 256;
    int64_t blocks = (total + threads - 1) / threads;
    const int64_t cap = (int64_t)dbl::sm_count() * 16;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    resize_kernel<Tin, Tout, 8><<<(int)blocks, threads, 0, s>>>(static_cast<const Tin*>(in), static_cast<Tout*>(out),
                                                                n, hi, wi, c, ho, wo, cs);
    return dbl::launch_check("progressive_resize launch");
}

// The stem's unrolled input.  Position (n, m, q) holds rg source rows
// y = rg*m + e - pad_h (e < rg), each as 8 column taps x (8/rg) channels:
// element (e, t, ch) is the resized pixel at (y, q*sw + t - pw), channel ch
// (zero outside the image, for t >= taps and for ch >= c).
// One CTA per unrolled row (n, m): it interpolates the rg resized rows once
// into shared memory (with pw zero columns on each side), each pixel rounded
// to the storage format there, then writes the row's Q positions as 16-byte
// chunks (8 elements), consecutive threads on consecutive chunks, each chunk
// one 16-byte shared-memory load of two staged pixels (a tap pair) or of one
// (8 channels).  Staging fp32 values and rounding every copy of a pixel in the
// write phase issued twice the instructions there, with 8.7-way bank
// conflicts.  A resolution equal to the source's (lambda = 0, i0 = j: the
// interpolation returns the pixel itself, bit for bit) skips the taps.
constexpr int kStemMaxW = 1024;  // widest resized row a CTA stages (host-checked)
// Threads per CTA.  A CTA's two phases are short chains of dependent memory operations, so
// the kernel is bound by how many rows are in flight: 64-thread CTAs (32 per SM) measured
// 177 us for 224 -> 224 at batch 512 against 242 us with 256-thread CTAs (8 per SM).
constexpr int kStemThreads = 64;

// Per-channel affine map of 8-bit pixels to the network's input values,
// x = p*scale + bias, rounded after the product and after the sum (no
// contraction: the same bits as the same two fp32 operations on the host).
struct PixelNorm {
    float scale[8], bias[8];
};

template <typename Tin>
__device__ __forceinline__ float stem_pixel(const Tin* p, int ch, const PixelNorm& nm);
template <>
__device__ __forceinline__ float stem_pixel<float>(const float* p, int ch, const PixelNorm&)
{
    return __ldg(p);
}
template <>
__device__ __forceinline__ float stem_pixel<uint8_t>(const uint8_t* p, int ch, const PixelNorm& nm)
{
    return __fadd_rn(__fmul_rn((float)__ldg(p), nm.scale[ch]), nm.bias[ch]);
}


// Bilinear value from the four taps (a, b) on the upper source row and (c, d) on the lower one:
// (1-l)*p + l*q as one rounded product (l*q) and one fused multiply-add, written out so that the
// bits do not depend on how the compiler contracts the expression.
__device__ __forceinline__ float lerp_rn(float p, float q, float l) { return __fmaf_rn(1.f - l, p, __fmul_rn(l, q)); }
__device__ __forceinline__ float bilerp(float a, float b, float c, float d, float lx, float ly)
{
    return lerp_rn(lerp_rn(a, b, lx), lerp_rn(c, d, lx), ly);
}

// Staged row width in pixels: the resized row with pw zero columns on each side and 8 more for
// the taps past its end, rounded up to an even count so that pixel pairs start on 16 bytes.
__host__ __device__ __forceinline__ int32_t stem_staged_width(int32_t wo, int32_t pw) { return (wo + 2 * pw + 9) & ~1; }

template <int RG, typename Tin>
__global__ void __launch_bounds__(kStemThreads) resize_stem_kernel(const Tin* __restrict__ in, act_t* __restrict__ out,
                                                          int32_t hi, int32_t wi, int32_t c, int32_t ho, int32_t wo,
                                                          int32_t M, int32_t Q, int32_t taps, int32_t sw, int32_t pw,
                                                          int32_t ph, const PixelNorm nm)
{
    dbl::dev::grid_dependency_trigger();  // a convolution launched next may start its set-up
    constexpr int32_t cu = 8 / RG;  // channels per tap
    // staged rows: [RG][wst][cu] in the storage format (cu*2 bytes per pixel), column x at index x + pw
    extern __shared__ __align__(16) uint8_t staged[];
    const int32_t wst = stem_staged_width(wo, pw);
    const int32_t m = blockIdx.x % M, b = blockIdx.x / M;
    const Tin* base = in + (int64_t)b * hi * wi * c;
    const bool ident = hi == ho && wi == wo;
    // the RG source rows of this unrolled row: taps once per CTA
    Taps ty[RG];
    bool yin[RG];
#pragma unroll
    for (int e = 0; e < RG; ++e) {
        const int32_t y = RG * m + e - ph;
        yin[e] = y >= 0 && y < ho;
        ty[e] = axis_taps(yin[e] ? y : 0, hi, ho);
    }
    // one staged column (its RG pixels, all channels) per thread and iteration: the column taps
    // once for the RG rows, each pixel rounded to the storage format once (not once per copy)
    for (int32_t xs = threadIdx.x; xs < wst; xs += blockDim.x) {
        const int32_t x = xs - pw;
        const bool in_x = x >= 0 && x < wo;
        const Taps tx = axis_taps(in_x && !ident ? x : 0, wi, wo);
#pragma unroll
        for (int e = 0; e < RG; ++e) {
            float v[cu];
#pragma unroll
            for (int ch = 0; ch < cu; ++ch) v[ch] = 0.f;
            if (yin[e] && in_x) {
                if (ident) {
                    const Tin* p = base + ((int64_t)ty[e].i0 * wi + x) * c;
#pragma unroll
                    for (int ch = 0; ch < cu; ++ch)
                        if (ch < c) v[ch] = stem_pixel(p + ch, ch, nm);
                } else {
                    const Tin* r0 = base + (int64_t)ty[e].i0 * wi * c;
                    const Tin* r1 = base + (int64_t)ty[e].i1 * wi * c;
#pragma unroll
                    for (int ch = 0; ch < cu; ++ch)
                        if (ch < c)
                            v[ch] = bilerp(stem_pixel(r0 + tx.i0 * c + ch, ch, nm),
                                           stem_pixel(r0 + tx.i1 * c + ch, ch, nm),
                                           stem_pixel(r1 + tx.i0 * c + ch, ch, nm),
                                           stem_pixel(r1 + tx.i1 * c + ch, ch, nm), tx.lam, ty[e].lam);
                }
            }
            act2_t h[cu / 2];
#pragma unroll
            for (int k = 0; k < cu / 2; ++k) h[k] = dbl::act::pack2(v[2 * k], v[2 * k + 1]);
            uint8_t* dst = staged + ((size_t)e * wst + xs) * cu * 2;
            if constexpr (cu == 4)
                *reinterpret_cast<uint2*>(dst) = *reinterpret_cast<const uint2*>(h);
            else
                *reinterpret_cast<uint4*>(dst) = *reinterpret_cast<const uint4*>(h);
        }
    }
    __syncthreads();
    // the unrolled row: 16-byte chunks gathered from the staged pixels, consecutive threads on
    // consecutive chunks; a chunk is 16 staged bytes (two pixels of one row, or one of 8 channels)
    uint4* orow = reinterpret_cast<uint4*>(out) + ((int64_t)b * M + m) * Q * 8;
    const uint4 zero = make_uint4(0u, 0u, 0u, 0u);  // +0 in every lane of either format
    const bool pairs16 = (sw & 1) == 0;  // pixel pairs q*sw + t0 (t0 even) start on 16 bytes
    for (int32_t idx = threadIdx.x; idx < Q * 8; idx += blockDim.x) {
        const int32_t q = idx >> 3, chunk = idx & 7;
        uint4 val;
        if constexpr (RG == 2) {
            // chunk = (row e, tap pair): taps t0, t0+1 of 4 channels each
            const int32_t e = chunk >> 2, t0 = (chunk & 3) * 2;
            const uint8_t* pp = staged + ((size_t)e * wst + q * sw + t0) * 8;
            if (pairs16) {
                val = *reinterpret_cast<const uint4*>(pp);
            } else {
                const uint2 lo = *reinterpret_cast<const uint2*>(pp), hi2 = *reinterpret_cast<const uint2*>(pp + 8);
                val = make_uint4(lo.x, lo.y, hi2.x, hi2.y);
            }
            if (t0 >= taps) val = zero;
            if (t0 + 1 >= taps) val.z = val.w = 0u;
        } else {
            // chunk = tap t of 8 channels
            val = chunk < taps ? *reinterpret_cast<const uint4*>(staged + ((size_t)q * sw + chunk) * 16) : zero;
        }
        orow[idx] = val;
    }
}

}  // namespace

namespace {

template <typename Tin>
int resize_stem_impl(const Tin* in, int32_t n, int32_t h_in, int32_t w_in, int32_t c, const PixelNorm& nm, void* out,
                     int32_t h_out, int32_t w_out, int32_t taps, int32_t stride_w, int32_t pad_w, int32_t row_group,
                     int32_t pad_h, int32_t rows_out, void* stream)
{
    using namespace dbl;
    if (!in || !out || n < 0 || h_in <= 0 || w_in <= 0 || c <= 0 || h_out <= 0 || w_out <= 0 || taps <= 0 ||
        stride_w <= 0 || pad_w < 0 || pad_h < 0 || rows_out <= 0)
        return set_error(DBL_ERR_INVALID, "progressive_resize_stem: bad sizes or null pointer");
    if (row_group != 1 && row_group != 2)
        return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize_stem: row_group must be 1 or 2");
    if (c > 8 / row_group || taps > 8)
        return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize_stem: at most 8 taps and 8/row_group channels");
    if (h_out > h_in || w_out > w_in) return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize_stem: upsampling");
    if (h_in > 16384 || w_in > 16384) return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize_stem: input side above 16384");
    if (!aligned16(out)) return set_error(DBL_ERR_INVALID, "progressive_resize_stem: output must be 16-byte aligned");
    const int32_t Q = (w_out + 2 * pad_w - taps) / stride_w + 1;
    if (Q <= 0) return set_error(DBL_ERR_INVALID, "progressive_resize_stem: empty output");
    if ((int64_t)n * rows_out >= (int64_t)1 << 31 || (int64_t)Q * 8 >= (int64_t)1 << 31)
        return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize_stem: output too large for 32-bit indexing");
    if (w_out + 2 * pad_w + 8 > kStemMaxW + 16 || (Q - 1) * stride_w + 8 > w_out + 2 * pad_w + 8)
        return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize_stem: rows wider than %d pixels", kStemMaxW);
    if (n == 0) return DBL_OK;
    const int blocks = n * rows_out;  // one CTA per unrolled row
    const size_t smem = (size_t)stem_staged_width(w_out, pad_w) * 8 * sizeof(act_t);  // rg rows x 8/rg channels
    if (row_group == 2)
        resize_stem_kernel<2, Tin><<<blocks, kStemThreads, smem, as_stream(stream)>>>(
            in, static_cast<act_t*>(out), h_in, w_in, c, h_out, w_out, rows_out, Q, taps, stride_w, pad_w, pad_h,
            nm);
    else
        resize_stem_kernel<1, Tin><<<blocks, kStemThreads, smem, as_stream(stream)>>>(
            in, static_cast<act_t*>(out), h_in, w_in, c, h_out, w_out, rows_out, Q, taps, stride_w, pad_w, pad_h,
            nm);
    return launch_check("progressive_resize_stem launch");
}

}  // namespace

extern "C" int dbl_progressive_resize_stem(const float* in, int32_t n, int32_t h_in, int32_t w_in, int32_t c, void* out,
                                           int32_t h_out, int32_t w_out, int32_t taps, int32_t stride_w, int32_t pad_w,
                                           int32_t row_group, int32_t pad_h, int32_t rows_out, void* stream)
{
    const PixelNorm nm{};
    return resize_stem_impl(in, n, h_in, w_in, c, nm, out, h_out, w_out, taps, stride_w, pad_w, row_group, pad_h,
                            rows_out, stream);
}

extern "C" int dbl_progressive_resize_stem_u8(const uint8_t* in, int32_t n, int32_t h_in, int32_t w_in, int32_t c,
                                              const float* scale, const float* bias, void* out, int32_t h_out,
                                              int32_t w_out, int32_t taps, int32_t stride_w, int32_t pad_w,
                                              int32_t row_group, int32_t pad_h, int32_t rows_out, void* stream)
{
    using namespace dbl;
    if (!scale || !bias) return set_error(DBL_ERR_INVALID, "progressive_resize_stem_u8: null scale or bias");
    if (c <= 0 || c > 8) return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize_stem_u8: 1..8 channels");
    PixelNorm nm{};
    for (int ch = 0; ch < c; ++ch) {
        nm.scale[ch] = scale[ch];
        nm.bias[ch] = bias[ch];
    }
    return resize_stem_impl(in, n, h_in, w_in, c, nm, out, h_out, w_out, taps, stride_w, pad_w, row_group, pad_h,
                            rows_out, stream);
}

extern "C" int dbl_progressive_resize(const void* in, int in_dtype, int32_t n, int32_t h_in, int32_t w_in, int32_t c,
                                      void* out, int out_dtype, int32_t h_out, int32_t w_out, int32_t c_out_stride,
                                      void* stream)
{
    using namespace dbl;
    if (!in || !out || n < 0 || h_in <= 0 || w_in <= 0 || c <= 0 || h_out <= 0 || w_out <= 0)
        return set_error(DBL_ERR_INVALID, "progressive_resize: bad sizes or null pointer");
    if (c > 8 || c_out_stride < c || c_out_stride > 8)
        return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize: supports 1..8 channels, stride c..8");
    if (h_in > 16384 || w_in > 16384)
        return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize: input side above 16384");
    if (h_out > h_in || w_out > w_in)
        return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize: upsampling %dx%d -> %dx%d", h_in, w_in, h_out,
                         w_out);
    if ((in_dtype != DBL_F32 && in_dtype != DBL_BF16) || (out_dtype != DBL_F32 && out_dtype != DBL_BF16))
        return set_error(DBL_ERR_INVALID, "progressive_resize: dtype must be DBL_F32 or DBL_BF16");
    if (!aligned16(out)) return set_error(DBL_ERR_INVALID, "progressive_resize: output must be 16-byte aligned");
    if ((int64_t)n * h_out * w_out >= (int64_t)1 << 31)
        return set_error(DBL_ERR_UNSUPPORTED, "progressive_resize: output too large for 32-bit indexing");
    if (n == 0) return DBL_OK;
    cudaStream_t s = as_stream(stream);
    if (in_dtype == DBL_F32 && out_dtype == DBL_BF16)
        return launch_resize<float, act_t>(in, out, n, h_in, w_in, c, h_out, w_out, c_out_stride, s);
    if (in_dtype == DBL_F32 && out_dtype == DBL_F32)
        return launch_resize<float, float>(in, out, n, h_in, w_in, c, h_out, w_out, c_out_stride, s);
    if (in_dtype == DBL_BF16 && out_dtype == DBL_BF16)
        return launch_resize<act_t, act_t>(in, out, n, h_in, w_in, c, h_out, w_out, c_out_stride, s);
    return launch_resize<act_t, float>(in, out, n, h_in, w_in, c, h_out, w_out, c_out_stride, s);
}
