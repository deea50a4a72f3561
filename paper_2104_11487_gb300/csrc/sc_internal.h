// Internal declarations of the Skip-Conv CUDA library (not part of the ABI).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "skipconv.h"

namespace sc {

// Device error word values (written by kernels, read by the host).
enum : int { DEV_OK = 0, DEV_TIMEOUT = 1, DEV_BAD_INDEX = 2 };

struct Layer {
    skipconv_params p;
    int ho, wo, nby, nbx;
    int cpg, opg;           // input / output channels per group
    int esize;              // bytes per element of dtype
    int path;               // SKIPCONV_PATH_CUDA_CORE or SKIPCONV_PATH_TENSOR_CORE
    int num_sms;
    int device;
    cudaStream_t stream;
    float gate_thr;         // threshold on the raw local l1 sum S (see api)

    // device state
    void* xbuf[2];          // ping-pong x_{t-1} / x_{t-2} frames, dtype
    uint8_t* chg[2];        // per input pixel: x_t != x_{t-1}, for the last two steps
    float* pix_l1;          // per input pixel: sum over channels of |r| (scratch)
    float* pix_taps;        // Gumbel gate: per input pixel and tap, sum_c phi[tap][c] r[c] (scratch)
    float* gphi;            // Gumbel gate function phi, [k_h*k_w][c_in] float32
    float gphi_bias;
    int gphi_set;           // 1 once skipconv_set_gate_weights was called
    uint8_t* mask;          // [n][nby][nbx]
    int32_t* list;          // active block ids
    int32_t* counters;      // [0], [1]: active-block count of even / odd steps
    float* z;               // [n][ho][wo][c_out]
    void* y;                // [n][ho][wo][c_out] dtype or NULL
    float* bias;            // [c_out]
    float* w_cc;            // [k_h][k_w][cpg][c_out] fp32 (CUDA-core path)
    __nv_bfloat16* w_tc;    // [co_pad][k_h*k_w*ci_pad] bf16 (tensor-core path)
    int ci_pad, co_pad;     // tensor-core padding of c_in (multiple of 64) and c_out (of 128)
    void* x_stage;          // device staging frame for skipconv_step_host (lazy)
    // skipconv_step_host_async (lazy): staging frames of x and z, copy streams, and per slot the events
    // "x uploaded", "x consumed by the step", "z staged", "z downloaded"
    void* xs_async[2];
    float* zs_async[2];
    cudaStream_t up_stream, down_stream;
    cudaEvent_t ev_up[2], ev_used[2], ev_zready[2], ev_down[2];
    long long async_steps;
    size_t state_bytes;

    // error word: pinned, mapped host memory
    int* err_host;
    int* err_dev;
    int* open_hint_host;    // fused step: the last sparse step's open-block count, written by the kernel into
    int* open_hint_dev;     // mapped host memory (same allocation as err_host); picks the next launch's form

    // profiling (host): launch counts per kernel kind, optional event pairs
    long long launches[SKIPCONV_PROFILE_KINDS];
    int prof_on;
    int prof_n, prof_cap;
    cudaEvent_t* prof_ev;   // 2 * prof_cap events
    int* prof_kind;
    double prof_ms[SKIPCONV_PROFILE_KINDS];

    // recurrence bookkeeping (host)
    long long t;            // steps since reset (selects the ping-pong buffers)
    int key;                // next step is a key frame
    long long since_key;    // steps since the last key frame, that one included

    // tensor-core path: prebuilt TMA descriptors of the two x_{t-1} buffers and the weights
    int tc_x5d;             // 1: halo tiles as one 5-D TMA box per channel chunk; 0: 4-D boxes per 8 channels
    CUtensorMap tmap_xbuf[2];
    CUtensorMap tmap_w;
    int tc_ws;              // 1: use the weight-stationary kernel
    CUtensorMap tmap_xrow[2];  // weight-stationary kernel: 128-byte-row halo boxes of the state frames
    int tc_z_tma;           // 1: the z tensor map below is valid (c_out multiple of 4)
    CUtensorMap tmap_z;

    // fused step kernel (sc_step_fused.cu)
    int fused;              // 1: the step is one cooperative tensor-core launch; 2: one CUDA-core launch
    int* sched;             // fused step: grid abort flag (16 ints reserved)
    uint64_t* pnorm;        // fused step: per pixel (epoch << 32) | fp32 norm
    uint32_t* gtag;         // fused step: per gate block (epoch << 1) | open
    uint32_t epoch;         // fused step: tag of the last launched step

    // one-launch CUDA-core step (sc_step_local.cu)
    int local_staged;       // 1: its TMA-footprint / staged-weight form
    int local_tc;           // 1: the staged form's contraction runs on the tensor cores (tcgen05)
    CUtensorMap tmap_fp[2]; // footprint boxes of the two state frames
    CUtensorMap tmap_ztile; // tile boxes of z
    void* w_loc;            // weights packed per CTA slice, layer dtype
    uint8_t* ychg;          // per gate block: the last step may have changed y (layers with y)
    uint8_t* tile_chg;      // [2][tiles]: some owned input pixel's change flag is set in chg[parity]
    int ntiles;             // tiles of the staged form
    int local_resident;     // CTAs of the staged form that fit on the GPU at once (SMs x CTAs per SM)

    // stack propagation (skipconv_link_inputs): the layers whose y this layer takes as x_t and as
    // the shortcut, and their step counts when this layer last stepped
    struct Layer* link_x;
    struct Layer* link_sc;
    long long link_x_seen, link_sc_seen;
    long long steps;        // steps since create (never reset)
    float* z_prev;          // warped steps: the second z buffer (the warp writes it, then the two swap)
    float* tx;              // warped steps on the staged form: T(x_{t-1}) in fp32 (allocated at the first one)
    CUtensorMap tmap_tx;    //   and its footprint boxes
};

// ------------------------------------------------------------------ launchers
// Active-block count of the step being enqueued (step t uses slot t % 2; the
// gate of step t clears slot (t+1) % 2 for the next step).
inline int32_t* step_count(const Layer& L) { return L.counters + (L.t & 1); }
inline int32_t* next_count(const Layer& L) { return L.counters + ((L.t + 1) & 1); }

// Gate (sc_gate.cu): pass 1, residual norms per pixel and the state commit;
// pass 2, block gates and the open-block list (a programmatic dependent of pass 1)
cudaError_t launch_gate_pixels(const Layer& L, const void* x_t, const void* x_prev, void* x_next,
                               const uint8_t* chg_prev, uint8_t* chg_cur, int force);
cudaError_t launch_gate_blocks(const Layer& L, int force);
// The Gumbel gate's two passes (Eq. 8): per-pixel tap products, then per-block f and threshold
size_t gumbel_smem_bytes(const Layer& L);
// Shared-memory limits of the Gumbel passes (at create)
cudaError_t gumbel_prepare(const Layer& L);
cudaError_t launch_gate_pixels_gumbel(const Layer& L, const void* x_t, const void* x_prev, void* x_next,
                                      const uint8_t* chg_prev, uint8_t* chg_cur);
cudaError_t launch_gate_blocks_gumbel(const Layer& L, int force);

// CUDA-core convolution and elementwise kernels (sc_conv_cc.cu)
cudaError_t launch_conv_cc(const Layer& L, const void* x_t, const void* x_prev);
cudaError_t launch_y_refresh(const Layer& L, const void* shortcut);
cudaError_t launch_reset_z(const Layer& L);
// The step's open blocks of z (count, ids, [b][b][c_out] values) into device-addressable buffers
// (mapped host memory for skipconv_step_host_sparse_async).
cudaError_t launch_gather_open_blocks(const Layer& L, const int32_t* count, float* zb, int32_t* list_out,
                                      int32_t* count_out);
cudaError_t launch_pack_weights(Layer& L, const void* w_oihw, double* w_l1_out);

// Tensor-core convolution (sc_conv_tc.cu)
bool conv_tc_supported(const skipconv_params& p, const char** why);
cudaError_t conv_tc_prepare(Layer& L);     // tensor maps of the state buffers and weights
cudaError_t launch_conv_tc(const Layer& L, const void* x_t, const void* x_prev, int prev_index);

// Weight-stationary tensor-core convolution (sc_conv_ws.cu), for layers that keep no y
bool conv_ws_supported(const Layer& L);
cudaError_t conv_ws_prepare(Layer& L);
cudaError_t launch_conv_ws(const Layer& L, const void* x_t, int prev_index);

// Fused step (sc_step_fused.cu): gate passes 1-2 and the weight-stationary
// convolution in one persistent cooperative launch, pipelined over streams.
bool step_fused_supported(const Layer& L);
cudaError_t step_fused_prepare(Layer& L);
cudaError_t launch_step_fused(Layer& L, const void* x_t, int force);

// One-launch step for CUDA-core layers (sc_step_local.cu): a CTA per tile of
// gate blocks computes residual, norms, gates, convolution, y and the commit
// from its own input footprint.
constexpr size_t LOCAL_MAX_SMEM = 226 * 1024;
// Layers whose dense step is at most this many MACs run on this form under
// SKIPCONV_PATH_AUTO even where tensor cores could serve them: at that size a
// step is bound by latency (a few memory round trips), not by arithmetic.
constexpr double LOCAL_AUTO_MAX_MACS = 67108864.0;   // 2^26
bool step_local_preferred(const Layer& L);
bool step_local_supported(const Layer& L);
// Warped residuals (Eq. 10-11) run on this step (the staged form's warped variant, else the general
// form): the layer must keep the frame size.
bool step_local_warp_supported(const Layer& L);
cudaError_t step_local_prepare(Layer& L);
// px / psc: the linked producers of x_t / of the shortcut whose y-change flags
// are valid for this step (NULL: not linked, or not valid for this step).
cudaError_t launch_step_local(Layer& L, const void* x_t, const void* shortcut, int force, const Layer* px,
                              const Layer* psc, const float* flow = nullptr);
// Warped residual (Eq. 10-11), before launch_step_local with the same flow: warps z~ into the second z
// buffer, which becomes z (y = act of it without a shortcut), and, where the staged form's warped
// variant runs, writes T(x_{t-1}) in fp32 and commits x_t with the change flags.
cudaError_t launch_step_warp_pass(Layer& L, const void* x_t, const void* shortcut, const float* flow);

// Driver entry point for tensor-map encoding (resolved once through the runtime).
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_tiled_fn();

void set_error(const char* fmt, ...);
// Raise (never lower) a kernel's dynamic shared-memory limit to `bytes`.
cudaError_t ensure_dynamic_smem(const void* func, size_t bytes);
// Host-side check of a parameter block (sizes, enums, limits); sets the error text.
int validate(const skipconv_params* p);

}  // namespace sc

// ------------------------------------------------------------- device helpers
namespace sc {

__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

__device__ __forceinline__ float activate(float v, int act)
{
    if (act == SKIPCONV_ACT_RELU) return v > 0.f ? v : 0.f;
    if (act == SKIPCONV_ACT_SILU) return v / (1.f + expf(-v));
    return v;
}

}  // namespace sc
