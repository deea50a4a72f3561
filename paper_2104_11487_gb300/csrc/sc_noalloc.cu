// skipconv_gate_noalloc: the block gate of one frame pair (residual, channel
// l1 norm, support sum, block maximum, threshold, compact list) computed
// without any allocation.
//
// Who needs it: callers that must not allocate device memory at step time.
// A process that has handed the device's memory to a caching allocator (as a
// PyTorch server does) can see cudaMalloc fail or force the cache to shrink,
// and cudaMalloc/cudaFree synchronise the whole device, which a latency-bound
// caller cannot afford.  A handle (skipconv_create) allocates its state once;
// this entry point needs no handle: its only scratch (the per-pixel norms and
// the open-block counter) is a file-scope __device__ array of fixed size that
// is part of the library's module image.
//
// Set-up: the first call on a device, with that device current, looks the
// scratch up with cudaGetSymbolAddress (this is where the CUDA runtime loads
// the module, and with it the array, on that device) and caches the address
// per device; later calls only launch.  Make that first call before any
// stream capture.  The scratch is shared by every call on a device: calls
// whose work can overlap on the device (different streams, or different host
// threads) race on it and must be serialised by the caller.
#include <mutex>

#include "sc_internal.h"

namespace sc {
namespace {

constexpr int kCounterBytes = 256;  // open-block counter, padded to keep the norms 256-byte aligned

// [0, 256): int32 open-block counter, zeroed by pass 1 of every call.
// [256, 256 + 4 * SKIPCONV_NOALLOC_MAX_PIXELS): float32 l1 norm of r per input pixel.
static __device__ __align__(256) unsigned char g_gate_scratch[kCounterBytes + 4 * SKIPCONV_NOALLOC_MAX_PIXELS];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_ptr[kMaxDevices];

struct NoallocGeom {
    int n, H, W, Ho, Wo, KH, KW, stride, pad, b, nby, nbx;
};

__device__ __forceinline__ float chunk_l1(const uint4& a, const uint4& b, __nv_bfloat16*)
{
    const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
    const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b);
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 fa = __bfloat1622float2(pa[k]);
        const float2 fb = __bfloat1622float2(pb[k]);
        s += fabsf(fa.x - fb.x) + fabsf(fa.y - fb.y);
    }
    return s;
}

__device__ __forceinline__ float chunk_l1(const uint4& a, const uint4& b, float*)
{
    float s = fabsf(__uint_as_float(a.x) - __uint_as_float(b.x));
    s += fabsf(__uint_as_float(a.y) - __uint_as_float(b.y));
    s += fabsf(__uint_as_float(a.z) - __uint_as_float(b.z));
    s += fabsf(__uint_as_float(a.w) - __uint_as_float(b.w));
    return s;
}

// Pass 1: sum_c |x_t - x_prev| per input pixel (Eq. 5's channel part, p = 1).
// G lanes share a pixel; with `vec` each lane reads 16-byte chunks, otherwise
// single elements.  Block 0 zeroes the counter that pass 2 appends with.
template <typename T>
__global__ void __launch_bounds__(256) noalloc_pixel_norm_kernel(const T* __restrict__ xt, const T* __restrict__ xp,
                                                                 float* __restrict__ norm, int32_t* __restrict__ count,
                                                                 long long n_pix, int C, int vec, int log2g)
{
    if (blockIdx.x == 0 && threadIdx.x == 0) *count = 0;
    const int lane = threadIdx.x & 31;
    const int G = 1 << log2g;
    const int sub = lane & (G - 1);
    const int gpw = 32 >> log2g;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    const int units = vec ? C * (int)sizeof(T) / 16 : C;
    for (long long base = warp * gpw; base < n_pix; base += nwarps * gpw) {
        const long long pix = base + (lane >> log2g);
        float s = 0.f;
        if (pix < n_pix) {
            for (int c = sub; c < units; c += G) {
                if (vec) {
                    const uint4 a = __ldg(reinterpret_cast<const uint4*>(xt) + pix * units + c);
                    const uint4 b = __ldg(reinterpret_cast<const uint4*>(xp) + pix * units + c);
                    s += chunk_l1(a, b, (T*)nullptr);
                } else {
                    s += fabsf(to_f32(xt[pix * C + c]) - to_f32(xp[pix * C + c]));
                }
            }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1)
            if (off < G) s += __shfl_xor_sync(0xffffffffu, s, off);
        if (pix < n_pix && sub == 0) norm[pix] = s;
    }
}

// Pass 2: one warp per b x b gate block: the largest support sum of the
// pixel norms over the block's output locations (Eq. 5 over the k_h x k_w
// receptive field with stride and zero padding; block max-pooling of Sec. 3.2)
// against the threshold; open blocks are appended to the list with one atomic
// per eight blocks.
__global__ void __launch_bounds__(256) noalloc_block_gate_kernel(const float* __restrict__ norm,
                                                                 uint8_t* __restrict__ mask,
                                                                 int32_t* __restrict__ list,
                                                                 int32_t* __restrict__ count, NoallocGeom g,
                                                                 float thr, int force)
{
    __shared__ int flags[8];
    const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long nblocks = (long long)g.n * g.nby * g.nbx;
    const long long blk = (long long)blockIdx.x * 8 + wid;
    int open = 0;
    if (blk < nblocks) {
        if (force) {
            open = 1;
        } else {
            const int bx = (int)(blk % g.nbx);
            const long long rest = blk / g.nbx;
            const int by = (int)(rest % g.nby);
            const int nn = (int)(rest / g.nby);
            const float* Pn = norm + (size_t)nn * g.H * g.W;
            const int bh = min(g.b, g.Ho - by * g.b), bw = min(g.b, g.Wo - bx * g.b);
            const int fy0 = by * g.b * g.stride - g.pad, fx0 = bx * g.b * g.stride - g.pad;
            float best = -1.f;
            for (int q = lane; q < bh * bw; q += 32) {
                const int i = q / bw, j = q - (q / bw) * bw;
                float S = 0.f;
                for (int kh = 0; kh < g.KH; ++kh) {
                    const int yy = fy0 + i * g.stride + kh;
                    if (yy < 0 || yy >= g.H) continue;
                    for (int kw = 0; kw < g.KW; ++kw) {
                        const int xx = fx0 + j * g.stride + kw;
                        if (xx < 0 || xx >= g.W) continue;
                        S += Pn[(size_t)yy * g.W + xx];
                    }
                }
                best = fmaxf(best, S);
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, off));
            open = best > thr ? 1 : 0;
        }
        if (lane == 0) mask[blk] = (uint8_t)open;
    }
    if (lane == 0) flags[wid] = open;
    __syncthreads();
    if (wid == 0) {
        const int f = lane < 8 ? flags[lane] : 0;
        const unsigned bal = __ballot_sync(0xffffffffu, f);
        int base = 0;
        if (lane == 0 && bal) base = atomicAdd(count, __popc(bal));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (f) list[base + __popc(bal & ((1u << lane) - 1u))] = (int32_t)(blockIdx.x * 8 + lane);
    }
}

// Address of the scratch on the current device (set-up on first use).
cudaError_t scratch_on_current_device(unsigned char** out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_gate_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_ptr[dev] = p;
    }
    *out = static_cast<unsigned char*>(g_scratch_ptr[dev]);
    return cudaSuccess;
}

}  // namespace
}  // namespace sc

using namespace sc;

extern "C" SKIPCONV_API int skipconv_gate_noalloc(const skipconv_params* params, const void* x_t, const void* x_prev,
                                                  uint8_t* block_mask, int32_t* active_list, int32_t* active_count,
                                                  void* stream)
{
    const int st = validate(params);
    if (st != SKIPCONV_OK) return st;
    const skipconv_params& p = *params;
    if (!x_t || !x_prev || !block_mask || !active_list || !active_count)
        return set_error("skipconv_gate_noalloc: NULL pointer argument"), SKIPCONV_ERR_INVALID;
    if (p.gate == SKIPCONV_GATE_OUTPUT || p.gate == SKIPCONV_GATE_GUMBEL)
        return set_error("skipconv_gate_noalloc: the output-norm and Gumbel gates need weights; use a layer handle"),
               SKIPCONV_ERR_UNSUPPORTED;
    const long long n_pix = (long long)p.n_streams * p.h * p.w;
    if (n_pix > SKIPCONV_NOALLOC_MAX_PIXELS)
        return set_error("skipconv_gate_noalloc: n_streams*h*w = %lld exceeds the static scratch of %d pixels",
                         n_pix, (int)SKIPCONV_NOALLOC_MAX_PIXELS),
               SKIPCONV_ERR_INVALID;

    unsigned char* scratch = nullptr;
    cudaError_t e = scratch_on_current_device(&scratch);
    if (e != cudaSuccess) {
        set_error("skipconv_gate_noalloc: scratch set-up failed: CUDA error %d: %s", (int)e, cudaGetErrorString(e));
        return SKIPCONV_ERR_CUDA;
    }
    int32_t* count = reinterpret_cast<int32_t*>(scratch);
    float* norm = reinterpret_cast<float*>(scratch + kCounterBytes);
    cudaStream_t s = static_cast<cudaStream_t>(stream);

    const int es = p.dtype == SKIPCONV_BF16 ? 2 : 4;
    const int vec = ((p.c_in * es) % 16 == 0) && ((uintptr_t)x_t % 16 == 0) && ((uintptr_t)x_prev % 16 == 0);
    const int units = vec ? p.c_in * es / 16 : p.c_in;
    int log2g = 0;
    while ((1 << log2g) < units && log2g < 5) ++log2g;
    const long long gpw = 32 >> log2g;
    const long long ctas = ((n_pix + gpw - 1) / gpw + 7) / 8;
    int dev = 0, sms = 0;
    e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) {
        set_error("CUDA error %d: %s", (int)e, cudaGetErrorString(e));
        return SKIPCONV_ERR_CUDA;
    }
    const long long cap = (long long)sms * 8;
    const int grid1 = (int)(ctas < cap ? (ctas > 0 ? ctas : 1) : cap);
    if (p.dtype == SKIPCONV_BF16)
        noalloc_pixel_norm_kernel<__nv_bfloat16><<<grid1, 256, 0, s>>>(
            (const __nv_bfloat16*)x_t, (const __nv_bfloat16*)x_prev, norm, count, n_pix, p.c_in, vec, log2g);
    else
        noalloc_pixel_norm_kernel<float><<<grid1, 256, 0, s>>>((const float*)x_t, (const float*)x_prev, norm, count,
                                                               n_pix, p.c_in, vec, log2g);

    NoallocGeom g;
    g.n = p.n_streams; g.H = p.h; g.W = p.w;
    g.Ho = (p.h + 2 * p.pad - p.k_h) / p.stride + 1;
    g.Wo = (p.w + 2 * p.pad - p.k_w) / p.stride + 1;
    g.KH = p.k_h; g.KW = p.k_w; g.stride = p.stride; g.pad = p.pad; g.b = p.block;
    g.nby = (g.Ho + p.block - 1) / p.block;
    g.nbx = (g.Wo + p.block - 1) / p.block;
    const double thr = p.gate == SKIPCONV_GATE_INPUT_MEAN ? (double)p.eps * p.c_in * p.k_h * p.k_w : (double)p.eps;
    const long long nblocks = (long long)g.n * g.nby * g.nbx;
    noalloc_block_gate_kernel<<<(unsigned)((nblocks + 7) / 8), 256, 0, s>>>(norm, block_mask, active_list, count, g,
                                                                            (float)thr, p.dense_mode ? 1 : 0);
    e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaMemcpyAsync(active_count, count, sizeof(int32_t), cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) {
        set_error("CUDA error %d: %s", (int)e, cudaGetErrorString(e));
        return SKIPCONV_ERR_CUDA;
    }
    return SKIPCONV_OK;
}
