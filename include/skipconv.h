/*
 * skipconv.h — C ABI of the GB300 (sm_103a) Skip-Convolution layer step.
 *
 * Method: Habibian et al., "Skip-Convolutions for Efficient Video Processing",
 * CVPR 2021 (arXiv 2104.11487).  One handle is one Skip-Conv layer applied to
 * n_streams independent video streams.  It keeps, per stream, the previous
 * input x_{t-1} and the output state z~_{t-1}, and each step computes
 *
 *     r_t   = x_t - x_{t-1}                                   (Eq. 2)
 *     g     = block gate of the local l1 norm of r_t           (Eq. 5 / Eq. 7,
 *             b x b blocks by max-pooling, Sec. 3.2 "Structured Sparsity")
 *     z~_t  = z~_{t-1} + g (.) (w * r_t)                       (Eq. 3)
 *
 * convolving only inside open blocks; closed blocks keep z~_{t-1} untouched.
 * The first step after create/reset is a key frame (Sec. 3.1: r_1 = x_1,
 * computed over the whole frame).
 *
 * Layouts (all row-major, no padding between rows):
 *   frames x_t, x_{t-1}, shortcut, y : [n_streams][h][w][c]        (NHWC)
 *   z                                 : [n_streams][ho][wo][c_out] float32
 *   weights                           : [c_out][c_in/groups][k_h][k_w] (OIHW)
 *   block mask                        : [n_streams][nby][nbx] uint8
 *   active list                       : int32 block ids (n*nby + by)*nbx + bx
 * with ho = (h + 2*pad - k_h)/stride + 1, wo likewise, nby = ceil(ho/block),
 * nbx = ceil(wo/block).  Element type of x, shortcut, weights and y is
 * `dtype` (float32 or bfloat16); z is always float32; bias is float32.
 *
 * Execution: every call enqueues work on the CUDA stream given at create and
 * returns without waiting, except where a function says it synchronises.
 * Pointers marked "device" must be device-accessible and stay valid until the
 * enqueued work has completed (stream order).  All functions return a
 * skipconv_status; no function throws.  A kernel that detects an internal
 * failure (for example a wait that ran out) records a device error word; the
 * next ABI call on that handle returns SKIPCONV_ERR_DEVICE.
 *
 * Threading: a handle must not be used from two host threads at once.
 * Different handles are independent.
 */
#ifndef SKIPCONV_H
#define SKIPCONV_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SKIPCONV_API __attribute__((visibility("default")))
#else
#define SKIPCONV_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct skipconv_s* skipconv_handle;

typedef enum {
    SKIPCONV_OK = 0,
    SKIPCONV_ERR_INVALID = -1,     /* bad argument, shape or handle            */
    SKIPCONV_ERR_UNSUPPORTED = -2, /* valid request this build does not cover  */
    SKIPCONV_ERR_CUDA = -3,        /* a CUDA runtime or driver call failed     */
    SKIPCONV_ERR_OOM = -4,         /* device or pinned-host allocation failed  */
    SKIPCONV_ERR_TIMEOUT = -5,     /* a bounded device wait ran out            */
    SKIPCONV_ERR_DEVICE = -6       /* a kernel recorded an internal error      */
} skipconv_status;

typedef enum {
    SKIPCONV_GATE_INPUT_MEAN = 0,  /* Eq. 5, l1 norm / (c_in*k_h*k_w) > eps    */
    SKIPCONV_GATE_INPUT_SUM = 1,   /* Eq. 5, l1 norm > eps                     */
    SKIPCONV_GATE_OUTPUT = 2,      /* Eq. 7, ||w||_1 * l1 norm > eps            */
    SKIPCONV_GATE_GUMBEL = 3       /* Eq. 8 at inference: f(r; phi) > eps, f a
                                      one-output-channel conv of r with the layer's
                                      kernel, stride and padding (eps = 0 is
                                      round(sigmoid(f))); phi from
                                      skipconv_set_gate_weights; k_h*k_w <= 9    */
} skipconv_gate;

typedef enum { SKIPCONV_F32 = 0, SKIPCONV_BF16 = 1 } skipconv_dtype;

typedef enum { SKIPCONV_ACT_NONE = 0, SKIPCONV_ACT_RELU = 1, SKIPCONV_ACT_SILU = 2 } skipconv_act;

typedef enum {
    SKIPCONV_PATH_AUTO = 0,        /* tensor cores where supported, else CUDA cores;
                                      layers whose dense step is at most 2^26 MACs
                                      run the one-launch step, a CTA per tile of
                                      gate blocks (a step of that size is latency-
                                      bound), with its contraction on the tensor
                                      cores for dense (groups = 1) bf16 layers    */
    SKIPCONV_PATH_CUDA_CORE = 1,   /* float32 FMA direct convolution              */
    SKIPCONV_PATH_TENSOR_CORE = 2, /* tcgen05 implicit GEMM (bf16 in, fp32 accum)  */
    SKIPCONV_PATH_TENSOR_CORE_SEPARATE = 3, /* the same convolution, but never fused with
                                      the gate: three launches per step           */
    SKIPCONV_PATH_CUDA_CORE_SEPARATE = 4 /* the CUDA-core convolution in its own launch
                                      after the two gate passes (CUDA_CORE runs the
                                      whole step as one launch where it can)      */
} skipconv_path;

typedef struct {
    int n_streams;     /* independent streams advanced together, >= 1              */
    int c_in, c_out;   /* channels; both divisible by groups                       */
    int h, w;          /* input frame size                                          */
    int k_h, k_w;      /* kernel size                                               */
    int stride;        /* >= 1, both directions                                     */
    int pad;           /* zero padding, both directions, >= 0                       */
    int groups;        /* 1 = dense, c_in = c_out = groups: depthwise               */
    int block;         /* b: gate block edge on the output grid, >= 1               */
    float eps;         /* gate threshold, >= 0                                      */
    int gate;          /* skipconv_gate                                             */
    int dtype;         /* skipconv_dtype of x, shortcut, weights and y              */
    int activation;    /* skipconv_act applied to y only (z is pre-activation)      */
    int emit_y;        /* 1: keep y = act(z [+ shortcut]) in dtype for the next layer */
    int dense_mode;    /* 1: every gate open (in-library dense reference)           */
    int conv_path;     /* skipconv_path                                             */
    int key_interval;  /* > 0: every key_interval-th step after a key frame is a key
                          frame again (Table 4's periodic reset: x_{t-1} = 0,
                          z = bias, whole frame); 0: only after create or reset */
} skipconv_params;

/* Create a layer.  Copies and repacks the weights (device pointer, OIHW,
 * dtype), copies the optional bias (device float32 [c_out], NULL = 0),
 * allocates all state on the current device and resets it (next step is a key
 * frame).  `stream` is a cudaStream_t (NULL = legacy default stream).
 * Synchronises the stream once.  On failure *out is NULL.
 * Errors: INVALID (NULL pointer, non-positive or inconsistent sizes, unknown
 * enum), UNSUPPORTED (conv_path forced to a path that cannot run this shape),
 * OOM, CUDA. */
SKIPCONV_API int skipconv_create(const skipconv_params* params, const void* weights_oihw,
                    const float* bias, void* stream, skipconv_handle* out);

/* Reset the recurrence (Sec. 3.1 key frame; Table 4's reference-frame reset):
 * x_{t-1} = 0, z = bias, and the next step processes the whole frame.
 * Enqueued on the handle's stream. */
SKIPCONV_API int skipconv_reset_state(skipconv_handle h);

/* One Skip-Conv step (Eq. 2, 5/7, 3); a key frame when the handle was just
 * created or reset, or when params.key_interval steps have passed since the
 * last key frame (then the reset is enqueued first).  x_t: device frame [n][h][w][c_in] in
 * dtype, 16-byte aligned.  shortcut: NULL, or a device tensor
 * [n][ho][wo][c_out] in dtype added to z before the activation when y is
 * kept (then y is refreshed over the whole frame).  Updates z in place at the
 * open blocks, the gate outputs, y (if kept) and x_{t-1} <- x_t.  Enqueued;
 * x_t and shortcut must stay valid until the stream reaches this work. */
SKIPCONV_API int skipconv_step(skipconv_handle h, const void* x_t, const void* shortcut);

/* One step with a warped residual (Sec. 3.4, Eq. 10-11): the residual is
 * taken against the previous input warped by the flow, r_t = x_t - T(x_{t-1}),
 * and the previous output is warped the same way before the gated convolution
 * of r_t is added: z~_t = T~(z~_{t-1}) + g(r_t) (.) (w * r_t).  T samples at
 * (y + dy, x + dx) by bilinear interpolation of the four surrounding pixels,
 * a pixel outside the frame contributing zero; T~ does the same on the output
 * grid, so the layer must keep the frame size (stride 1, ho = h, wo = w).
 * flow: device float32 [n][h][w][2], (dy, dx) in pixels, 4-byte aligned.  A
 * key frame has no previous frame to warp and is the plain key-frame step.
 * Every location of z (and y) moves; the gate, list and x_{t-1} <- x_t are as
 * in skipconv_step.  The first warped step allocates a second z buffer (the
 * warp writes it and it becomes z, so the pointer skipconv_get_z returns
 * changes at every warped step) and, where the staged form runs, an fp32
 * frame for T(x_{t-1}).  Errors as skipconv_step, and UNSUPPORTED unless the
 * layer runs the one-launch CUDA-core step and keeps the frame size. */
SKIPCONV_API int skipconv_step_warped(skipconv_handle h, const void* x_t, const void* shortcut, const float* flow);

/* Stack propagation: the input of layer l+1 changes only where layer l's
 * output changed (the residual of Eq. 2 is zero elsewhere).  Declares that
 * this layer's x_t is producer_x's y and, if producer_sc is not NULL, that
 * its shortcut is producer_sc's y.  Every layer that keeps y publishes, per
 * gate block, whether its last step may have changed y (an open block, or a
 * changed shortcut).  At a step whose x_t (and shortcut) are those producers'
 * y and whose producers each stepped exactly once since this layer last did,
 * a tile whose footprint saw no such change, that committed no change at the
 * previous step and whose shortcut did not change, skips reading its inputs:
 * its residual is zero there, so the full step would keep every block closed
 * and write nothing.  Results are identical to unlinked steps.  Otherwise
 * (another x_t, a producer that stepped twice or not at all, key frames) the
 * step reads the whole frame as usual, and so does a layer whose tiles take at
 * most two waves of resident CTAs: skipping tiles takes no wave off such a
 * step, while reading the flags would delay every tile by a memory round
 * trip.  producer_x = NULL removes the links.
 * Errors: INVALID (NULL handle, self link, shortcut link without x link,
 * shapes, dtypes or streams that do not match), UNSUPPORTED (this layer not on
 * the one-launch CUDA-core step with TMA footprints, or a producer that keeps
 * no y or is not on the one-launch CUDA-core step).  Destroying a producer
 * drops the links to it; linking and destroying must not race with steps on
 * other threads. */
SKIPCONV_API int skipconv_link_inputs(skipconv_handle h, skipconv_handle producer_x, skipconv_handle producer_sc);

/* The same step on host buffers: copies x_t (host, [n][h][w][c_in] dtype;
 * pinned memory makes the copy asynchronous DMA) to the device, runs the
 * step, copies the whole z back to z_out (host float32 [n][ho][wo][c_out],
 * may be NULL to skip the read-back), and synchronises the stream before
 * returning.  The first call allocates a device staging frame. */
SKIPCONV_API int skipconv_step_host(skipconv_handle h, const void* x_t_host, float* z_out_host);

/* Pipelined host-buffer step: the same work as skipconv_step_host, enqueued
 * without waiting.  The copy of x_t_host (host, [n][h][w][c_in] dtype;
 * pinned memory, else the copy is synchronous) goes to one of two device
 * staging frames on the handle's upload stream; the step runs on the
 * handle's stream once that copy is done; z is then copied on the device to
 * one of two staging buffers and from there to z_out_host (host float32
 * [n][ho][wo][c_out], pinned; may be NULL) on the download stream.  So the
 * upload of step t+1 and the download of step t-1 overlap step t.  Both host
 * buffers are lent until skipconv_sync returns.  The first call allocates
 * the staging buffers (2 frames of x, 2 of z) and the two copy streams.
 * Errors: INVALID (NULL handle or x_t_host), OOM, CUDA; a device error word
 * set by an earlier step is reported as by skipconv_step. */
SKIPCONV_API int skipconv_step_host_async(skipconv_handle h, const void* x_t_host, float* z_out_host);

/* Pipelined host-buffer step with a sparse result (Eq. 3: z~ changes only at
 * the open blocks, the rest is copied from the previous step).  x_t_host is
 * uploaded and the step runs as in skipconv_step_host_async; then, on the
 * handle's stream, a kernel writes straight into the host buffers (pinned and
 * mapped into the device's address space, e.g. cudaHostAlloc; every pinned
 * allocation is mapped on systems with unified addressing):
 *   *count_host        the number of open blocks of this step;
 *   list_host[i]       the i-th open block id, (n * nby + by) * nbx + bx
 *                      (i < count; order unspecified, as skipconv_get_gate);
 *   z_blocks_host[i]   that block's z~ after the step, float32 [b][b][c_out]
 *                      (output locations past the frame's edge are 0).
 * A consumer that holds z~ applies the blocks to keep it equal to the
 * device's z~; after create, a reset or a key frame every block is open.
 * The buffers must have room for n*nby*nbx blocks and ids and are lent until
 * skipconv_sync returns.  Enqueued without waiting; the first call allocates
 * the two device staging frames of x (no staging of z).  Errors: INVALID
 * (NULL handle or pointer, or a host buffer the device cannot address), OOM,
 * CUDA; a device error word set by an earlier step is reported as by
 * skipconv_step. */
SKIPCONV_API int skipconv_step_host_sparse_async(skipconv_handle h, const void* x_t_host, float* z_blocks_host,
                                                 int32_t* list_host, int32_t* count_host);

/* Wait for every step and copy enqueued on the handle's streams; reports the
 * device error word (SKIPCONV_OK, SKIPCONV_ERR_TIMEOUT, SKIPCONV_ERR_DEVICE). */
SKIPCONV_API int skipconv_sync(skipconv_handle h);

/* The Gumbel gate's function (Eq. 8): phi_oihw, device float32
 * [1][c_in][k_h][k_w] (one output channel, the layer's kernel size), and its
 * bias.  Required before the first step of a SKIPCONV_GATE_GUMBEL layer; may
 * be called again to replace phi.  Copies phi (through the host) and
 * synchronises the stream.  Errors: INVALID (NULL handle or phi, a layer whose
 * gate is not GUMBEL), CUDA. */
SKIPCONV_API int skipconv_set_gate_weights(skipconv_handle h, const float* phi_oihw, float phi_bias);

/* Synchronise the stream and free everything.  NULL is accepted. */
SKIPCONV_API int skipconv_destroy(skipconv_handle h);

/* Read-only views of the handle's device state, valid until the next step,
 * reset or destroy (read them in stream order). */
SKIPCONV_API int skipconv_get_z(skipconv_handle h, const float** z);
SKIPCONV_API int skipconv_get_y(skipconv_handle h, const void** y);            /* NULL unless emit_y */
SKIPCONV_API int skipconv_get_prev_input(skipconv_handle h, const void** x_prev); /* x_{t-1} for the next step */
/* Gate of the last step: block mask, the compacted list of open block ids
 * (order unspecified) and its length (device int32). */
SKIPCONV_API int skipconv_get_gate(skipconv_handle h, const uint8_t** block_mask, const int32_t** active_list,
                      const int32_t** active_count);

/* Shape facts of a handle (host values). */
typedef struct {
    int ho, wo;        /* output frame size                                   */
    int nby, nbx;      /* gate blocks per stream                              */
    int conv_path;     /* where the contraction runs: SKIPCONV_PATH_CUDA_CORE or
                          SKIPCONV_PATH_TENSOR_CORE                           */
    int num_sms;       /* SMs of the device the handle lives on               */
    size_t state_bytes;/* device bytes held by the handle                     */
    int fused;         /* 0: separate launches (gate passes, convolution, y);
                          1: each step is one cooperative tensor-core launch
                          (gate and convolution pipelined over the streams);
                          2: each step is one launch, a CTA per tile of gate
                          blocks working from its own input footprint (its
                          contraction on tcgen05 where conv_path says so)     */
} skipconv_info;
SKIPCONV_API int skipconv_get_info(skipconv_handle h, skipconv_info* info);

/* Statistics of the last step.  Synchronises the stream.  active_blocks is
 * the number of open blocks over all streams, active_locations the output
 * locations inside them, macs = active_locations * c_out * (c_in/groups) *
 * k_h * k_w (the MAC count of Eq. 9's accounting).  Any pointer may be NULL. */
SKIPCONV_API int skipconv_get_stats(skipconv_handle h, long long* active_blocks, long long* active_locations,
                       double* macs);

/* Synchronise the stream and report the device error word:
 * SKIPCONV_OK, SKIPCONV_ERR_TIMEOUT or SKIPCONV_ERR_DEVICE. */
SKIPCONV_API int skipconv_check_device(skipconv_handle h);

/* Failure-detection self-test: launches, on the handle's stream, one kernel
 * whose bounded wait (the shared-memory barrier wait every pipelined kernel
 * of the library uses) is never satisfied.  It gives up after limit_ns
 * (1 .. 1e9) and records a timeout in the handle's device error word, as a
 * stuck step would; no memory is touched but that word.  Synchronises and
 * returns what skipconv_check_device then reports: SKIPCONV_ERR_TIMEOUT.
 * From then on the handle refuses work (steps and resets return the same
 * status) and is only fit for skipconv_destroy; the CUDA context and other
 * handles stay usable.  Errors: INVALID (NULL handle, limit out of range). */
SKIPCONV_API int skipconv_selftest_timeout(skipconv_handle h, long long limit_ns);

/* Per-kernel timing.  Kernel kinds: 0 gate_pixel (residual, channel l1 norm,
 * state commit), 1 gate_block (support norm, block gate, compaction), 2 the
 * convolution of the open blocks (either path), 3 y refresh, 4 the fused
 * tensor-core step (all of 0-2 in one launch), 5 the one-launch CUDA-core step
 * (all of 0-3), 6 the warp pass of skipconv_step_warped (z~ and, on the staged
 * form, x_{t-1}, Eq. 10-11).  Launch counts are always kept; with enable = 1
 * each launch is also bracketed by CUDA events on the handle's stream.
 * skipconv_profile resets both. */
#define SKIPCONV_PROFILE_KINDS 7
SKIPCONV_API int skipconv_profile(skipconv_handle h, int enable);
/* Synchronise the stream and report, per kernel kind (arrays of
 * SKIPCONV_PROFILE_KINDS), the launches and the summed event-timed
 * milliseconds since skipconv_profile (milliseconds are 0 unless timing was
 * enabled). */
SKIPCONV_API int skipconv_profile_read(skipconv_handle h, long long* launches, double* ms);

/* Largest n_streams*h*w that skipconv_gate_noalloc accepts: its static device
 * scratch holds one float32 norm per input pixel (4 MiB + 256 B per device). */
#define SKIPCONV_NOALLOC_MAX_PIXELS (1 << 20)

/* Block gate of one frame pair, with no allocation of any kind.  The paper has
 * no counterpart: this is a deployment form of the gate that skipconv_step
 * runs, for callers that must not allocate device memory while they run -- a
 * process whose device memory is held by a caching allocator (cudaMalloc may
 * fail there, or force the cache to shrink) and latency-bound callers that
 * cannot take the device-wide synchronisation of cudaMalloc/cudaFree.  It
 * needs no handle.  It computes the same block gate as skipconv_step: for the
 * difference r = x_t - x_prev, the sum of |r| over each output location's
 * c_in x k_h x k_w receptive field (stride and zero padding as in params),
 * the maximum of that sum over each b x b block of output locations, and opens
 * the blocks whose maximum exceeds the threshold of params->gate (INPUT_MEAN
 * or INPUT_SUM; dense_mode = 1 opens every block).  The convolution fields of
 * params are validated as for skipconv_create and otherwise unused.
 *   x_t, x_prev  : device frames [n][h][w][c_in] in dtype (read only)
 *   block_mask   : device uint8 [n][nby][nbx], written
 *   active_list  : device int32 with room for n*nby*nbx ids; the open block
 *                  ids, order unspecified
 *   active_count : device int32, the number of open blocks
 *   stream       : cudaStream_t (NULL = legacy default stream)
 * Enqueued on `stream`; returns without waiting.  Scratch: one static
 * __device__ array of 256 + 4*SKIPCONV_NOALLOC_MAX_PIXELS bytes per device.
 * The first call on a device (with that device current) performs the set-up:
 * it takes the array's address with cudaGetSymbolAddress, where the runtime
 * loads the library's module on that device, and caches it; make that first
 * call before any stream capture.  Later calls only launch kernels and one
 * 4-byte device-to-device copy.  The open-block counter in the scratch is
 * zeroed on the device by every call.  Every call on a device shares the one
 * scratch: calls whose work may overlap on the device (different streams or
 * host threads) race and must be serialised by the caller.
 * Errors: INVALID (NULL pointer, bad params, n_streams*h*w above
 * SKIPCONV_NOALLOC_MAX_PIXELS), UNSUPPORTED (gate OUTPUT, which needs ||w||_1
 * that only a handle holds), CUDA (set-up or launch failed). */
SKIPCONV_API int skipconv_gate_noalloc(const skipconv_params* params, const void* x_t, const void* x_prev,
                                       uint8_t* block_mask, int32_t* active_list, int32_t* active_count,
                                       void* stream);

/* Human-readable name of a status code (static string). */
SKIPCONV_API const char* skipconv_status_string(int status);

/* Detail of the last failure on the calling thread (static per thread). */
SKIPCONV_API const char* skipconv_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* SKIPCONV_H */
