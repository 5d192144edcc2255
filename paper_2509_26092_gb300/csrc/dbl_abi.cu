// dbl_abi.cu -- host-side parts of the C ABI: error text, device queries,
// driver entry points for tensor-map encoding, and the host helpers of the
// planner (Sec. 3.3-3.4) and of progressive resizing (Sec. 4.1).
#include <math.h>
#include <stdarg.h>
#include <stdio.h>

#include <atomic>
#include <mutex>

#include "dbl_internal.cuh"

namespace dbl {

static thread_local char g_err[512] = "";
static std::atomic<int64_t> g_launches{0};

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

int set_error(int code, const char* fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

int sm_count()
{
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 148;
    if (dev < 64 && cached[dev]) return cached[dev];
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
        (void)cudaGetLastError();
        return 148;  // no device answered: a nominal count, never cached
    }
    if (dev < 64) cached[dev] = n;
    return n;
}

static void* driver_entry(const char* name)
{
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion(name, &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
        return nullptr;
    return fn;
}

PFN_encodeTiled encode_tiled()
{
    static std::once_flag once;
    static PFN_encodeTiled fn = nullptr;
    std::call_once(once, [] { fn = reinterpret_cast<PFN_encodeTiled>(driver_entry("cuTensorMapEncodeTiled")); });
    return fn;
}

PFN_encodeIm2col encode_im2col()
{
    static std::once_flag once;
    static PFN_encodeIm2col fn = nullptr;
    std::call_once(once, [] { fn = reinterpret_cast<PFN_encodeIm2col>(driver_entry("cuTensorMapEncodeIm2col")); });
    return fn;
}

int current_context_id(unsigned long long* id)
{
    typedef CUresult (*PFN_ctxGetCurrent)(CUcontext*);
    typedef CUresult (*PFN_ctxGetId)(CUcontext, unsigned long long*);
    static std::once_flag once;
    static PFN_ctxGetCurrent get_current = nullptr;
    static PFN_ctxGetId get_id = nullptr;
    std::call_once(once, [] {
        get_current = reinterpret_cast<PFN_ctxGetCurrent>(driver_entry("cuCtxGetCurrent"));
        get_id = reinterpret_cast<PFN_ctxGetId>(driver_entry("cuCtxGetId"));
    });
    *id = 0;
    if (!get_current || !get_id) return set_error(DBL_ERR_CUDA, "driver entry points cuCtxGetCurrent/cuCtxGetId missing");
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS) return set_error(DBL_ERR_CUDA, "cuCtxGetCurrent failed");
    if (!ctx) return DBL_OK;
    if (get_id(ctx, id) != CUDA_SUCCESS) return set_error(DBL_ERR_CUDA, "cuCtxGetId failed");
    return DBL_OK;
}

}  // namespace dbl

extern "C" {

const char* dbl_last_error(void) { return dbl::g_err; }

int dbl_version(void) { return 100; /* 0.1.0 */ }

int64_t dbl_kernel_launches(void) { return dbl::g_launches.load(std::memory_order_relaxed); }

int dbl_resize_taps(int32_t in, int32_t out, int32_t* i0, int32_t* i1, float* lambda)
{
    if (in <= 0 || out <= 0 || !i0 || !i1 || !lambda) return dbl::set_error(DBL_ERR_INVALID, "resize_taps: bad args");
    if (out > in) return dbl::set_error(DBL_ERR_UNSUPPORTED, "resize_taps: upsampling (%d -> %d)", in, out);
    for (int32_t j = 0; j < out; ++j) {
        const int64_t num = (int64_t)(2 * j + 1) * in - out;  // >= 0 when out <= in
        const int64_t den = 2 * (int64_t)out;
        const int64_t a = num / den;
        i0[j] = (int32_t)a;
        i1[j] = (int32_t)(a + 1 < in ? a + 1 : in - 1);
        lambda[j] = (float)(num - a * den) / (float)den;
    }
    return DBL_OK;
}

double dbl_update_factor(double d_small, double d_large, int sqrt_scheme)
{
    if (!(d_large > 0.0)) return NAN;
    const double r = d_small / d_large;
    return sqrt_scheme ? sqrt(r) : r;
}

int dbl_plan(double k, double d, int32_t n_small, int32_t n_large, double a, double b, double batch_large,
             int sqrt_scheme, double* d_large, double* d_small, double* batch_small, double* f_small)
{
    if (n_small < 1 || n_large < 0 || !(d > 0) || !(k > 0) || !(batch_large > 0) || !d_large || !d_small ||
        !batch_small || !f_small)
        return dbl::set_error(DBL_ERR_INVALID, "plan: bad arguments");
    const int32_t n = n_small + n_large;
    const double dL = k * d / n;                      // Eq. 4
    const double dS = (d - n_large * dL) / n_small;   // Eq. 6
    const double den = (a + b / batch_large) * dL / dS - a;  // Eq. 8
    if (!(dS > 0) || !(den > 0)) return dbl::set_error(DBL_ERR_INVALID, "plan: no positive small batch");
    *d_large = dL;
    *d_small = dS;
    *batch_small = b / den;
    *f_small = dbl_update_factor(dS, dL, sqrt_scheme);
    return DBL_OK;
}

}  // extern "C"
