/*
 * dbl.h -- C ABI of libdbl.so: the GB300 (sm_103a) kernels of one training
 * step of the hybrid dual-batch / cyclic-progressive learning scheme
 * (arXiv 2509.26092) on ResNet-18.
 *
 * Conventions shared by every call
 * --------------------------------
 *  - Every call returns DBL_OK (0) or a negative DBL_ERR_* code; the text of
 *    the last error on the calling thread is available from dbl_last_error().
 *  - Device pointers are owned by the caller (PyTorch allocates them); the
 *    library never allocates or frees device memory.  Scratch space is passed
 *    in as `ws`/`ws_bytes`, sized by the matching *_workspace_bytes() call.
 *  - Work is enqueued on the caller's CUDA stream, passed as `void*`
 *    (a cudaStream_t; NULL is the legacy default stream).  No call
 *    synchronises the device or the stream, so calls can be captured into a
 *    CUDA graph.  Exceptions, marked "host" or "synchronous", are stated.
 *  - Tensors are dense row-major.  Activations are NHWC bfloat16, conv
 *    weights are KRSC, master weights and gradients are fp32.  Every tensor
 *    base address must be 16-byte aligned and every NHWC channel count a
 *    multiple of 8 (a 16-byte pixel row); violations return DBL_ERR_INVALID
 *    before anything is launched.  There is no slow fallback path.
 *  - Kernels that wait on an asynchronous copy give up after a bounded time,
 *    record DBL_ERR_TIMEOUT in a device-side status word and return; read it
 *    with dbl_device_status().
 *  - Storage format.  The library is built twice from the same sources, with
 *    the same entry points: libdbl.so stores activations, activation gradients
 *    and the convolutions' weight copies as bfloat16; libdbl_f16.so (built
 *    with DBL_ACT_F16) stores them as IEEE binary16, the format of the
 *    paper's mixed-precision ImageNet runs (Sec. 5.2.3), to be used with the
 *    loss scaling below.  Every parameter named *_bf16 (and DBL_BF16) denotes
 *    the library's 16-bit format; fp32 arguments are fp32 in both.  The
 *    tensor cores multiply the two operands in that one format (never mixed)
 *    and accumulate in fp32.
 */
#ifndef DBL_H
#define DBL_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define DBL_API __attribute__((visibility("default")))
#else
#define DBL_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

enum {
    DBL_OK = 0,
    DBL_ERR_INVALID = -1,     /* null pointer, misaligned, inconsistent shape        */
    DBL_ERR_UNSUPPORTED = -2, /* well-formed request outside what the kernels cover  */
    DBL_ERR_CUDA = -3,        /* a CUDA call or launch failed                        */
    DBL_ERR_TIMEOUT = -4,     /* a device-side wait gave up (see dbl_device_status)  */
    DBL_ERR_WORKSPACE = -5    /* ws_bytes smaller than *_workspace_bytes()           */
};

enum { DBL_F32 = 0, DBL_BF16 = 1 }; /* element types for dbl_progressive_resize */

/* Text of the last error raised on the calling thread ("" if none). Host. */
DBL_API const char* dbl_last_error(void);

/* Library version, major*10000 + minor*100 + patch.  Host. */
DBL_API int dbl_version(void);

/* Number of kernel launches this library has issued from the host since it
 * was loaded (all threads, all devices).  Launches replayed from a captured
 * CUDA graph are not counted again.  Host; for instrumentation. */
DBL_API int64_t dbl_kernel_launches(void);

/* Synchronous: reads and clears the device-side status word of the current
 * device (DBL_OK or DBL_ERR_TIMEOUT), after synchronising the device.  For
 * tests and diagnostics only; never call it inside a captured graph. */
DBL_API int dbl_device_status(int32_t* status);

/* ========================================================================
 * Convolution passes as implicit GEMM on the tensor cores.
 *
 * The ResNet-18 of the paper (Sec. 5.1.1) is built from these three passes;
 * the training step needs the forward pass and, through Eq. 1 (the gradient
 * of the batch-mean loss), the data and weight gradients.
 *
 *   y[n,p,q,k] = sum_{r,s,c} x[n, p*stride_h + r - pad_h, q*stride_w + s - pad_w, c] * w[k,r,s,c]
 *   P = (h + 2*pad_h - r)/stride_h + 1,  Q = (w + 2*pad_w - s)/stride_w + 1
 *
 * x: [n,h,w,c] bf16, w: [k,r,s,c] bf16, y: [n,P,Q,k] bf16, all NHWC/KRSC.
 * Supported: c and k multiples of 64 (any r, s <= 8 with stride <= 2 and
 * pad <= 3 per axis for the forward and weight passes; square filters with
 * equal strides and pads for the data gradient), or c == 8 (3 colour
 * channels zero-padded to 8) for the forward and weight passes.  The stem of
 * ResNet-18 is run as an r x 1 convolution over the input unrolled along W
 * (see dbl_progressive_resize_stem).
 *
 * Environment (read once per process): DBL_CONV_CTA_PAIRS=0 runs every pass on
 * single CTAs, =2 puts every 128/256-column tile on CTA pairs; DBL_CONV_PDL=1
 * launches the passes with programmatic stream serialization, so that a
 * kernel's set-up overlaps the end of the kernel before it on the stream
 * (faster with one stream of work, slower when another stream competes for
 * the SMs).  Neither changes what is computed.
 * ======================================================================== */

/* Host: overrides DBL_CONV_PDL for the convolution launches that follow, in
 * this process, from any thread: 1 = programmatic stream serialization on,
 * 0 = off, -1 = back to the environment's choice.  Launches already enqueued
 * (or captured) keep the attribute they were launched with. */
DBL_API int dbl_set_conv_pdl(int32_t mode);

/* Host, for tests of the bounded waits: arms the next implicit-GEMM
 * convolution launch (a pass that dbl_conv_plan reports as
 * DBL_KERNEL_IGEMM) of this process so that its thread block 0 never
 * issues the load of its first K-block.  That block's MMA issuer then waits
 * on a stage that never fills; the wait gives up after its limit (about 2 s),
 * records DBL_ERR_TIMEOUT in the device status (dbl_device_status), and every
 * role of the block winds down through its own bounded waits, letting the
 * copies it issued land before it returns.  The other blocks finish normally;
 * the launch's outputs are not valid.  No fault is raised and the context
 * stays usable.  Applies to one launch, then disarms itself. */
DBL_API int dbl_conv_test_stall_next(void);
typedef struct {
    int32_t n, h, w, c; /* input activation shape (NHWC)                    */
    int32_t k, r, s;    /* output channels and filter size (KRSC weights)   */
    int32_t stride, pad;       /* along H (and along W when stride_w == 0)   */
    int32_t stride_w, pad_w;   /* along W; stride_w == 0: same as stride/pad */
} dbl_conv_shape;

enum { DBL_PASS_FWD = 0, DBL_PASS_DGRAD = 1, DBL_PASS_WGRAD = 2 };

/* Bytes of scratch the given pass needs for this shape (0 if none).  Host. */
DBL_API size_t dbl_conv_workspace_bytes(const dbl_conv_shape* shape, int pass);

/* How a convolution pass runs on the current device, without launching it
 * (host): the kernel (implicit GEMM, the 3x3 stride-1 window kernel, or the
 * window weight gradient), output columns per tile, CTAs per MMA (2: a CTA
 * pair with M = 256 MMAs across two SMs), tiles of the persistent loop, the
 * split-K slices of a weight gradient or the phases of a stride-2 data
 * gradient (else 1), the CTAs launched, and the window kernels' dynamic shared
 * memory per CTA (0 for the implicit GEMM).  The pass functions make the same
 * plan.  Errors: DBL_ERR_INVALID (null info, bad pass), and the shape errors of
 * the pass functions. */
enum { DBL_KERNEL_IGEMM = 0, DBL_KERNEL_WINDOW = 1, DBL_KERNEL_WINDOW_WGRAD = 2 };
typedef struct {
    int32_t kernel;
    int32_t tile_cols;
    int32_t ctas_per_mma;
    int32_t tiles;
    int32_t zdim;
    int32_t grid;
    int64_t smem_bytes;
} dbl_conv_plan_info;

DBL_API int dbl_conv_plan(const dbl_conv_shape* shape, int pass, dbl_conv_plan_info* info);

/* Forward pass.  Writes y (bf16, rounded to nearest even from the fp32
 * accumulator).  If ch_sum/ch_sumsq are non-NULL, also writes the per-output-
 * channel sums of the stored (rounded) y and of its squares over all n*P*Q
 * rows, [k] fp32 each: the batch statistics BatchNorm needs in training
 * mode.  Overwrites ch_sum/ch_sumsq (no accumulation). */
DBL_API int dbl_conv_fwd(const dbl_conv_shape* shape, const void* x_bf16, const void* w_bf16, void* y_bf16,
                 float* ch_sum, float* ch_sumsq, void* ws, size_t ws_bytes, void* stream);

/* Forward pass that leaves the BatchNorm statistics as partial sums for
 * dbl_bn_relu_fused_parts to reduce (one kernel launch fewer per layer than
 * dbl_conv_fwd + dbl_bn_relu_fused).  Writes y as dbl_conv_fwd does, and into
 * parts ([*nparts][2][k] fp32, caller-owned, at least
 * dbl_conv_stats_parts_bytes(shape) bytes) the sums of the stored y and of its
 * squares over the rows each of *nparts thread blocks stored.  *nparts (host
 * memory) is set at call time; the same shape on the same device always gives
 * the same value. */
DBL_API size_t dbl_conv_stats_parts_bytes(const dbl_conv_shape* shape);
DBL_API int dbl_conv_fwd_parts(const dbl_conv_shape* shape, const void* x_bf16, const void* w_bf16, void* y_bf16,
                               float* parts, size_t parts_bytes, int32_t* nparts, void* stream);

/* Data gradient: dx = d(sum y*dy)/dx, the adjoint of the forward pass in its
 * input.  dy: [n,P,Q,k] bf16; dx: [n,h,w,c] bf16 (fully overwritten).
 * Supported for stride 1, and for stride 2 with even h and w. */
DBL_API int dbl_conv_dgrad(const dbl_conv_shape* shape, const void* dy_bf16, const void* w_bf16, void* dx_bf16, void* ws,
                   size_t ws_bytes, void* stream);

/* Data gradient of a downsampling ResNet-18 block input (Sec. 5.1.1): the
 * block's first convolution (shape, stride 2) and its 1x1 stride-2 pad-0
 * projection shortcut both read the same input x, so
 *   dx = dgrad(shape; dy, w) + dgrad(1x1/2; dy2, w2),
 * computed in one pass (the projection term reaches only the even rows and
 * columns of dx, where it is accumulated with the main term).
 * dy2: [n, h/2, w/2, k2] bf16, w2: [k2, 1, 1, c] bf16; k2 a multiple of 64.
 * Requires stride 2 and even h, w.  dx is fully overwritten. */
DBL_API int dbl_conv_dgrad_proj(const dbl_conv_shape* shape, const void* dy_bf16, const void* w_bf16, int32_t k2,
                                const void* dy2_bf16, const void* w2_bf16, void* dx_bf16, void* ws, size_t ws_bytes,
                                void* stream);

/* Weight gradient: dw[k,r,s,c] = sum_{n,p,q} dy[n,p,q,k] * x[n, p*stride+r-pad, q*stride+s-pad, c],
 * fp32 [k,r,s,c].  accumulate != 0 adds to dw instead of overwriting it.
 * The split over n*P*Q is reduced in a fixed order (deterministic). */
DBL_API int dbl_conv_wgrad(const dbl_conv_shape* shape, const void* x_bf16, const void* dy_bf16, float* dw_f32,
                   int accumulate, void* ws, size_t ws_bytes, void* stream);

/* ========================================================================
 * BatchNorm (training mode) + residual + ReLU, the non-convolution layers of
 * ResNet-18 (Sec. 5.1.1).
 *
 *   mean = ch_sum/count, var = ch_sumsq/count - mean^2 (biased),
 *   invstd = 1/sqrt(var + eps),
 *   out = [ReLU]( gamma*(y - mean)*invstd + beta [+ residual] )
 *
 * y, residual, out: [count, c] bf16 (NHWC flattened); gamma, beta, ch_sum,
 * ch_sumsq, save_mean, save_invstd: [c] fp32.  ReLU'(0) is taken as 0.
 * ======================================================================== */
typedef struct {
    int64_t count; /* rows: n*h*w                  */
    int32_t c;     /* channels, a multiple of 8    */
    float eps;     /* variance epsilon (1e-5)      */
    int32_t relu;  /* nonzero: apply ReLU          */
} dbl_bn_shape;

/* Per-channel sum and sum of squares of y over all rows, [c] fp32 each.
 * (dbl_conv_fwd already provides them for its own output.) */
DBL_API int dbl_bn_stats(const dbl_bn_shape* shape, const void* y_bf16, float* ch_sum, float* ch_sumsq, void* stream);

/* Normalise + affine + optional residual + optional ReLU; writes out (bf16)
 * and the batch mean and 1/sqrt(var+eps) used (needed by the backward). */
DBL_API int dbl_bn_relu_fused(const dbl_bn_shape* shape, const void* y_bf16, const float* ch_sum, const float* ch_sumsq,
                      const float* gamma, const float* beta, const void* residual_bf16 /* or NULL */,
                      void* out_bf16, float* save_mean, float* save_invstd, void* stream);

/* dbl_bn_relu_fused with the batch statistics given as the partial sums of
 * dbl_conv_fwd_parts (parts [nparts][2][c]); they are reduced in the same fixed
 * order as dbl_conv_fwd reduces them, so the result is bit-identical to
 * dbl_conv_fwd + dbl_bn_relu_fused. */
DBL_API int dbl_bn_relu_fused_parts(const dbl_bn_shape* shape, const void* y_bf16, const float* parts, int32_t nparts,
                                    const float* gamma, const float* beta, const void* residual_bf16 /* or NULL */,
                                    void* out_bf16, float* save_mean, float* save_invstd, void* stream);

/* Bytes of scratch dbl_bn_relu_fused_bwd needs.  Host. */
DBL_API size_t dbl_bn_workspace_bytes(const dbl_bn_shape* shape);

/* Backward of dbl_bn_relu_fused.  The incoming gradient is dout [+ dout2]
 * (a tensor read by two consumers, e.g. a block output feeding the next
 * block's convolution and its shortcut), masked by ReLU through out > 0 when
 * shape->relu is set:  g = (dout + dout2) * [out > 0].  Then
 *   dbeta = sum g, dgamma = sum g*xhat, xhat = (y - mean)*invstd,
 *   dy = gamma*invstd*(g - dbeta/count - xhat*dgamma/count),
 * and, if dresidual is non-NULL, dresidual = g (the residual branch's
 * gradient).  dy, dresidual: bf16 [count, c]; dgamma, dbeta: fp32 [c]
 * (overwritten).  The channel sums are reduced in a fixed order.
 * out_bf16 may be NULL (with shape->relu set) when the forward pass had no
 * residual: the mask is then recomputed from y exactly as dbl_bn_relu_fused
 * decided it, [y*scale + shift > 0] with scale = gamma*invstd and shift =
 * beta - mean*scale, which needs beta (otherwise beta may be NULL). */
DBL_API int dbl_bn_relu_fused_bwd(const dbl_bn_shape* shape, const void* dout_bf16, const void* dout2_bf16 /* or NULL */,
                          const void* y_bf16, const void* out_bf16 /* or NULL */, const float* gamma,
                          const float* beta /* or NULL */, const float* save_mean, const float* save_invstd,
                          void* dy_bf16, void* dresidual_bf16 /* or NULL */, float* dgamma, float* dbeta, void* ws,
                          size_t ws_bytes, void* stream);

/* Same computation as dbl_bn_relu_fused_bwd, for callers that cannot hand
 * the library a workspace: their memory comes from an allocator they do not
 * control (a host framework that owns every device allocation), or their
 * device-memory footprint must be fixed once the process has started.  The
 * paper has no counterpart; this is a property of the library, not of the
 * method.
 *
 * The scratch lives in one statically sized device array inside libdbl.so
 * (2.1 MB, held on every device that loads the library until the process
 * exits).  Limit: c <= DBL_BN_NOALLOC_MAX_C (512); larger c returns
 * DBL_ERR_UNSUPPORTED before anything is launched.  The first call in a CUDA
 * context looks up the array's device address (cudaGetSymbolAddress) with
 * that context current and caches it under the context's unique ID; a context
 * destroyed and created again (cudaDeviceReset) gets a new ID, so its first
 * call looks the address up again.  That lookup may load the library's
 * module, so it must not run inside a stream capture: a first call while the
 * stream is capturing returns DBL_ERR_INVALID and launches nothing; make one
 * call outside capture first.  No device memory is allocated or freed by any
 * call.  All calls share the one
 * array, so calls whose kernels overlap on the GPU (two streams, two host
 * threads) race on it; serialise them.  Nothing in the array needs to start
 * at zero: each call writes every element it later reads. */
#define DBL_BN_NOALLOC_MAX_C 512
DBL_API int dbl_bn_relu_fused_bwd_noalloc(const dbl_bn_shape* shape, const void* dout_bf16,
                                          const void* dout2_bf16 /* or NULL */, const void* y_bf16,
                                          const void* out_bf16, const float* gamma, const float* beta, const float* save_mean,
                                          const float* save_invstd, void* dy_bf16, void* dresidual_bf16 /* or NULL */,
                                          float* dgamma, float* dbeta, void* stream);

/* dbl_bn_relu_fused (no residual, relu set) followed by dbl_maxpool_fwd of
 * its output, without storing that output: y, argmax as from
 * dbl_maxpool_fwd of bf16(ReLU(x*scale + shift)), with the statistics
 * finalized from ch_sum/ch_sumsq exactly as dbl_bn_relu_fused does (it also
 * writes save_mean/save_invstd).  The ImageNet stem's BatchNorm + ReLU +
 * 3x3/2 max pool (ResNet-18, Sec. 5.1.1).  shape: count = n*h*w rows of c
 * channels; x: [n,h,w,c] bf16 (the BatchNorm input).  The backward pass
 * recomputes the ReLU mask from x (dbl_bn_relu_fused_bwd with out = NULL). */
DBL_API int dbl_bn_relu_maxpool_fwd(const dbl_bn_shape* shape, int32_t n, int32_t h, int32_t w, const void* x_bf16,
                                    const float* ch_sum, const float* ch_sumsq, const float* gamma, const float* beta,
                                    float* save_mean, float* save_invstd, void* y_bf16, uint8_t* argmax,
                                    void* stream);

/* ========================================================================
 * Stem max pooling (ImageNet ResNet-18): 3x3 window, stride 2, padding 1,
 * padding counted as -infinity.  x: [n,h,w,c] bf16, y: [n,P,Q,c] bf16,
 * argmax: [n,P,Q,c] uint8, the window index r*3+s of the first maximum in
 * row-major window order (the tie rule).  The backward routes each of
 * dy [+ dy2] to its argmax and sums what lands on each input: dx [n,h,w,c].
 * ======================================================================== */
DBL_API int dbl_maxpool_fwd(int32_t n, int32_t h, int32_t w, int32_t c, const void* x_bf16, void* y_bf16, uint8_t* argmax,
                    void* stream);
DBL_API int dbl_maxpool_bwd(int32_t n, int32_t h, int32_t w, int32_t c, const void* dy_bf16, const void* dy2_bf16,
                    const uint8_t* argmax, void* dx_bf16, void* stream);

/* ========================================================================
 * Head forward + backward in one call: global average pooling (the pooling
 * that makes the network resolution-agnostic, Sec. 6), one fully connected
 * layer (Sec. 5.1.1) and softmax cross-entropy averaged over the batch (the
 * 1/n of Eq. 1).
 *   feat[n,c] = mean_hw x,  logits = feat*fc_w^T + fc_b,
 *   loss = mean_n (logsumexp(logits_n) - logits_n[label_n]),
 *   dlogits = (softmax - onehot)/n,  dfc_w = dlogits^T feat,  dfc_b = sum_n dlogits,
 *   dx[n,i,c] = (dlogits*fc_w)[n,c] / hw.
 * x: [n,hw,c] bf16; fc_w: [classes,c] fp32; fc_b: [classes] fp32;
 * labels: [n] int32 in [0,classes); loss: one fp32 on the device;
 * dfc_w, dfc_b: fp32 (overwritten); dx: [n,hw,c] bf16.
 * ======================================================================== */
DBL_API size_t dbl_head_workspace_bytes(int32_t n, int32_t c, int32_t classes);
DBL_API int dbl_head_fwd_bwd(int32_t n, int32_t hw, int32_t c, int32_t classes, const void* x_bf16, const float* fc_w,
                     const float* fc_b, const int32_t* labels, float* loss, float* dfc_w, float* dfc_b, void* dx_bf16,
                     void* ws, size_t ws_bytes, void* stream);

/* Head with the options of the hybrid scheme's training step:
 *  - dropout of the pooled features before the FC layer.  Cyclic progressive
 *    learning raises the dropout rate d with the resolution of each sub-stage
 *    (Sec. 4.1; 0.1 / 0.2 / 0.3 in Tables 7 and 9).  Inverted dropout:
 *      featd[n,c] = feat[n,c] * keep[n,c] / (1 - d),
 *    logits, loss, dfc_w, dfc_b as dbl_head_fwd_bwd with featd in place of
 *    feat, and dx[n,i,c] = (dlogits*fc_w)[n,c] * keep[n,c] / (1 - d) / hw, with
 *    keep[n,c] the mask dbl_dropout_mask writes for the same (d, seed, *step).
 *    step: device pointer to one uint64 (8-byte aligned) read by the kernels;
 *    after the call's last kernel it is incremented by one on the stream, so
 *    consecutive calls (and replays of a captured graph) draw fresh masks.
 *    drop_rate = 0: no dropout (step may be NULL and is not touched);
 *    outside [0, 1): DBL_ERR_INVALID.
 *  - loss scaling for mixed-precision training (Sec. 5.2.3): loss_scale is a
 *    device pointer to one fp32 S read by the kernels (NULL: S = 1); the
 *    backward pass starts from dlogits = (softmax - onehot) * S/n, so dfc_w,
 *    dfc_b and dx (and every gradient computed from dx) are S times the
 *    loss's gradients.  loss is reported unscaled.
 * With drop_rate 0 and loss_scale NULL this is dbl_head_fwd_bwd exactly.
 * Workspace as dbl_head_fwd_bwd. */
typedef struct {
    float drop_rate;
    uint64_t seed;
    uint64_t* step;
    const float* loss_scale;
} dbl_head_opts;
DBL_API int dbl_head_fwd_bwd_ex(int32_t n, int32_t hw, int32_t c, int32_t classes, const void* x_bf16, const float* fc_w,
                                const float* fc_b, const int32_t* labels, const dbl_head_opts* opts, float* loss,
                                float* dfc_w, float* dfc_b, void* dx_bf16, void* ws, size_t ws_bytes, void* stream);

/* The dropout mask of dbl_head_fwd_bwd_ex: keep[n,c] (uint8, 1 = kept)
 * for n samples of c features (c a multiple of 4; keep 4-byte aligned).
 * Feature c of sample n takes word c % 4 of the Philox4x64-10 block (Salmon
 * et al., SC 2011) at counter (n*c/4 + c/4, *step, 0, 0) with key (seed, 0),
 * and is kept when the word's upper 32 bits are at least
 * floor(drop_rate * 2^32) (an integer comparison, so the mask is exact).
 * step is read on the device and not changed.  drop_rate = 0 keeps all. */
DBL_API int dbl_dropout_mask(int32_t n, int32_t c, float drop_rate, uint64_t seed, const uint64_t* step,
                             uint8_t* keep, void* stream);

/* ========================================================================
 * Parameter-server merge of the two workers' pushes (Sec. 3.4, with the SGD
 * of Eq. 1 and momentum).  Each push i brings its worker's batch-mean
 * gradient g_i, scaled by the model-update factor f_i (1 for the large-batch
 * worker; d_S/d_L or sqrt(d_S/d_L) for the small-batch worker):
 *     u <- momentum*u - lr*f_i*g_i ;  w <- w + u
 * order 0: large push then small push (ASP arrival order, Sec. 2.4);
 * order 1: small then large; order 2: one step on f_L*g_L + f_S*g_S.
 * A NULL gradient is a worker that did not push (both NULL is invalid).
 * w, u: fp32 [n], updated in place; w16_out (or NULL): bf16 copy of the new
 * w, the weights the workers pull for their next step.
 * ======================================================================== */
typedef struct {
    float lr, momentum, f_large, f_small;
    int32_t order;
} dbl_merge_params;

DBL_API int dbl_ps_dual_batch_merge(float* w, float* u, void* w16_out, const float* g_large, const float* g_small, int64_t n,
                            const dbl_merge_params* params, void* stream);

/* The merge under mixed precision with loss scaling (Micikevicius et al., the
 * method of the paper's fp16 runs, Sec. 5.2.3).  A worker that scaled its loss
 * by S_i pushes S_i * g_i; this merge divides each push by its scale
 * (scale_large / scale_small: device pointers to the fp32 scale each worker
 * used; required for each non-NULL push), then applies the update of
 * dbl_ps_dual_batch_merge.  If *found_inf (device int32) is non-zero, nothing
 * is written: w, u and w16 keep their values.  Scales are powers of two (the
 * dynamic scale below keeps them so), so the division is exact. */
DBL_API int dbl_ps_dual_batch_merge_scaled(float* w, float* u, void* w16_out, const float* g_large,
                                           const float* g_small, int64_t n, const dbl_merge_params* params,
                                           const float* scale_large, const float* scale_small,
                                           const int32_t* found_inf, void* stream);

/* Sets *found_inf (device int32) to 1 if any of g[0, n) (fp32, device, 16-byte
 * aligned) is infinite or NaN; never clears it. */
DBL_API int dbl_grads_finite(const float* g, int64_t n, int32_t* found_inf, void* stream);

/* Dynamic loss scale, in device memory (16 bytes).  After the merge of a step:
 * if found_inf, the scale halves, good_steps restarts at 0 and skipped counts
 * the skipped update; otherwise good_steps counts up, and the scale doubles
 * when it reaches growth_interval (then restarts).  found_inf is cleared.
 * One thread, stream ordered. */
typedef struct {
    float scale;
    int32_t good_steps;
    int32_t found_inf;
    int32_t skipped;
} dbl_loss_scale;
DBL_API int dbl_loss_scale_update(dbl_loss_scale* state, int32_t growth_interval, void* stream);

/* Late and missing pushes.  Under ASP the server applies each push as it
 * arrives and does not wait for a worker that has stopped (Sec. 2.4); a
 * missing push is merged as g = NULL above.  With the workers on streams,
 * "has pushed" means "the worker's step event has completed".
 *
 * dbl_event_wait (host): DBL_OK once the cudaEvent_t `event` has completed,
 * DBL_ERR_TIMEOUT if it has not after timeout_s seconds (polling
 * cudaEventQuery; nothing is enqueued and the device is not synchronised),
 * DBL_ERR_CUDA if the query fails.  An event never recorded counts as
 * complete, as for cudaEventQuery.
 *
 * dbl_hold: holds `stream` until the host writes a non-zero value to *flag
 * (host-pinned memory the device can read, 4-byte aligned), or until
 * timeout_s (in (0, 10] s) has passed, whichever comes first; then writes
 * DBL_OK (released) or DBL_ERR_TIMEOUT (gave up) to *status (device or
 * pinned memory, may be NULL).  It emulates a worker whose push is delayed,
 * as a straggler on the paper's network would be; the wait is bounded, so
 * the stream always moves on.  Not a step of the method. */
DBL_API int dbl_event_wait(void* event, double timeout_s);
DBL_API int dbl_hold(const uint32_t* flag, double timeout_s, int32_t* status, void* stream);

/* ========================================================================
 * Progressive resizing for the low-resolution sub-stages of cyclic
 * progressive learning (Sec. 4.1): bilinear, half-pixel centres, no
 * antialiasing, downsampling only.  Output j of an axis reads source
 * i0 = floor(num/den), i1 = min(i0+1, in-1), weight lambda = (num - i0*den)/den
 * with num = (2j+1)*in - out, den = 2*out, all in exact integers.
 * in: [n,h_in,w_in,c] (DBL_F32 or DBL_BF16); out: [n,h_out,w_out,c_out_stride]
 * (DBL_F32 or DBL_BF16) with channels c..c_out_stride-1 set to zero.
 * h_out == h_in is a plain cast/pad; h_out > h_in is DBL_ERR_UNSUPPORTED.
 * ======================================================================== */
DBL_API int dbl_progressive_resize(const void* in, int in_dtype, int32_t n, int32_t h_in, int32_t w_in, int32_t c, void* out,
                           int out_dtype, int32_t h_out, int32_t w_out, int32_t c_out_stride, void* stream);

/* The same resize, written in the layout the tensor-core stem consumes.
 * Output position (n, m, q), m < rows_out, q < Q, holds row_group source rows
 * y = row_group*m + e - pad_h (e < row_group) of the resized image, each
 * unrolled along W for a stem with `taps` filter columns, column stride
 * stride_w and padding pad_w: element (e, t, ch) is the resized pixel at
 * (y, q*stride_w + t - pad_w), channel ch, for t = 0..7 and ch < 8/row_group
 * (zero outside the image, for t >= taps and for ch >= c):
 *   out[n][m][q][e][t][ch], bf16, 128 bytes per position,
 *   Q = (w_out + 2*pad_w - taps)/stride_w + 1.
 * With row_group 1 and pad_h 0 (rows_out = h_out), a taps x taps stem of
 * stride s equals an r x 1 convolution of this tensor (stride s along H
 * only, the stem's padding along H, 64 channels) with the weights stored as
 * [k][r][8][8]; with row_group 2 (a stride-2 stem: pad_h = its padding and
 * rows_out = P + ceil(r/2) - 1 for P output rows), it equals a ceil(r/2) x 1
 * valid convolution of stride 1 with the weights stored as [k][2*ceil(r/2)][8][4]
 * (rows r.. of that layout are not filter rows and must stay zero: their
 * weight gradient is not part of the method, see dbl_zero_f32_2d).
 * in: [n,h_in,w_in,c] fp32, c <= 8/row_group, taps <= 8. */
DBL_API int dbl_progressive_resize_stem(const float* in, int32_t n, int32_t h_in, int32_t w_in, int32_t c, void* out,
                                        int32_t h_out, int32_t w_out, int32_t taps, int32_t stride_w, int32_t pad_w,
                                        int32_t row_group, int32_t pad_h, int32_t rows_out, void* stream);

/* The same, from 8-bit pixels: in is [n,h_in,w_in,c] uint8 and the value the
 * resize sees is p*scale[ch] + bias[ch] (fp32, rounded after the product and
 * after the sum), the usual per-channel standardization of decoded images.
 * scale, bias: host arrays [c], read during the call. */
DBL_API int dbl_progressive_resize_stem_u8(const uint8_t* in, int32_t n, int32_t h_in, int32_t w_in, int32_t c,
                                           const float* scale, const float* bias, void* out, int32_t h_out,
                                           int32_t w_out, int32_t taps, int32_t stride_w, int32_t pad_w,
                                           int32_t row_group, int32_t pad_h, int32_t rows_out, void* stream);

/* Sets base[i*ld + j] = 0 for i < rows, j < cols (fp32, device memory, stream
 * ordered).  The ResNet-18 stem uses it to keep the weight gradient of the
 * padding rows of its row-grouped weight layout at zero, so that those
 * weights stay zero through the parameter-server update.  Not a step of the
 * paper's method. */
DBL_API int dbl_zero_f32_2d(float* base, int64_t rows, int64_t cols, int64_t ld, void* stream);

/* Host: the integer taps above for one axis (i0, i1, lambda: [out] each). */
DBL_API int dbl_resize_taps(int32_t in, int32_t out, int32_t* i0, int32_t* i1, float* lambda);

/* ========================================================================
 * Host-side planner of dual-batch learning (Sec. 3.3-3.4).
 * ======================================================================== */
/* Model-update factor of a small-batch worker: d_S/d_L, or sqrt(d_S/d_L)
 * when sqrt_scheme != 0 (Sec. 3.4).  Returns NaN for d_large <= 0. */
DBL_API double dbl_update_factor(double d_small, double d_large, int sqrt_scheme);

/* Eqs. 4-8: given the extra-time ratio k > 1, data amount d, worker counts,
 * the time-model coefficients a, b (per-batch time a*x + b, Eq. 2) and the
 * large batch B_L, returns d_L = k*d/n, d_S = (d - n_L*d_L)/n_S,
 * B_S = b/((a + b/B_L)*d_L/d_S - a) and f_S = d_S/d_L (scheme 1) or its root.
 * DBL_ERR_INVALID if n_small < 1 or the inputs give no positive B_S. */
DBL_API int dbl_plan(double k, double d, int32_t n_small, int32_t n_large, double a, double b, double batch_large,
             int sqrt_scheme, double* d_large, double* d_small, double* batch_small, double* f_small);

#ifdef __cplusplus
}
#endif
#endif /* DBL_H */
