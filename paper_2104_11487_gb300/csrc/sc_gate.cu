// Gate kernels of the Skip-Conv step.
//
// gate_pixel : one pass over x_t and x_{t-1} (the two full-frame reads of the
//              step).  Per input pixel it forms the residual r_t = x_t - x_{t-1}
//              (Eq. 2), its l1 norm over all input channels (the channel part of
//              the Input-Norm gate, Eq. 5, p = 1), and whether the pixel changed
//              bit-wise.  It also commits x_t into the ping-pong buffer that
//              becomes x_{t-1} at the next step, writing only pixels that
//              changed at this step or the previous one (every other pixel of
//              that buffer already holds x_t).
// gate_block : one warp per b x b output block.  Per output location it sums
//              the per-pixel l1 norms over the k_h x k_w receptive field (stride,
//              zero padding) — the local support norm of Eq. 5 — takes the
//              block maximum (max-pooling of the gate, Sec. 3.2) and compares it
//              with the threshold; open blocks are appended to a compact list
//              with one atomic per CTA.
#include "sc_internal.h"

namespace sc {
namespace {

__device__ __forceinline__ float l1_diff(const uint4& a, const uint4& b, __nv_bfloat16*)
{
    const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
    const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b);
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        float2 fa = __bfloat1622float2(pa[k]);
        float2 fb = __bfloat1622float2(pb[k]);
        s += fabsf(fa.x - fb.x) + fabsf(fa.y - fb.y);
    }
    return s;
}

__device__ __forceinline__ float l1_diff(const uint4& a, const uint4& b, float*)
{
    float s = fabsf(__uint_as_float(a.x) - __uint_as_float(b.x));
    s += fabsf(__uint_as_float(a.y) - __uint_as_float(b.y));
    s += fabsf(__uint_as_float(a.z) - __uint_as_float(b.z));
    s += fabsf(__uint_as_float(a.w) - __uint_as_float(b.w));
    return s;
}

__device__ __forceinline__ unsigned bits_differ(const uint4& a, const uint4& b)
{
    return (a.x ^ b.x) | (a.y ^ b.y) | (a.z ^ b.z) | (a.w ^ b.w);
}

// 16-byte vector path: a pixel's channels are `cpp` 16-byte chunks, handled
// by a group of G = 2^log2g lanes (each lane up to PER chunks).  Each warp
// iteration covers U consecutive groups of pixels so that 2*U*PER loads per
// lane are in flight before the first reduction.
template <typename T, int PER, int U>
__global__ void __launch_bounds__(256) gate_pixel_vec_kernel(
    const uint4* __restrict__ xt, const uint4* __restrict__ xp, uint4* __restrict__ xn,
    const uint8_t* __restrict__ chg_prev, uint8_t* __restrict__ chg_cur, float* __restrict__ pix_l1,
    long long n_pix, int cpp, int log2g, int32_t* __restrict__ counters)
{
    if (blockIdx.x == 0 && threadIdx.x == 0) counters[0] = 0;  // reset the active-block count
    const int lane = threadIdx.x & 31;
    const int G = 1 << log2g;
    const int sub = lane & (G - 1);
    const int gpw = 32 >> log2g;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long base = warp * gpw * U; base < n_pix; base += nwarps * gpw * U) {
        uint4 a[U][PER], b[U][PER];
#pragma unroll
        for (int v = 0; v < U; ++v) {
            const long long pix = base + v * gpw + (lane >> log2g);
#pragma unroll
            for (int k = 0; k < PER; ++k) {
                const int c = sub + k * G;
                if (pix < n_pix && c < cpp) {
                    a[v][k] = __ldg(xt + pix * cpp + c);
                    b[v][k] = __ldg(xp + pix * cpp + c);
                } else {
                    a[v][k] = make_uint4(0, 0, 0, 0);
                    b[v][k] = make_uint4(0, 0, 0, 0);
                }
            }
        }
#pragma unroll
        for (int v = 0; v < U; ++v) {
            const long long pix = base + v * gpw + (lane >> log2g);
            float s = 0.f;
            unsigned diff = 0;
#pragma unroll
            for (int k = 0; k < PER; ++k) {
                s += l1_diff(a[v][k], b[v][k], (T*)nullptr);
                diff |= bits_differ(a[v][k], b[v][k]);
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                if (off < G) {
                    s += __shfl_xor_sync(0xffffffffu, s, off);
                    diff |= __shfl_xor_sync(0xffffffffu, diff, off);
                }
            }
            if (pix < n_pix) {
                if (diff || chg_prev[pix]) {
#pragma unroll
                    for (int k = 0; k < PER; ++k) {
                        const int c = sub + k * G;
                        if (c < cpp) xn[pix * cpp + c] = a[v][k];
                    }
                }
                if (sub == 0) {
                    pix_l1[pix] = s;
                    chg_cur[pix] = diff ? 1 : 0;
                }
            }
        }
    }
}

// Element path for channel counts whose pixel is not a multiple of 16 bytes.
template <typename T, int PER>
__global__ void __launch_bounds__(256) gate_pixel_elem_kernel(
    const T* __restrict__ xt, const T* __restrict__ xp, T* __restrict__ xn,
    const uint8_t* __restrict__ chg_prev, uint8_t* __restrict__ chg_cur, float* __restrict__ pix_l1,
    long long n_pix, int C, int log2g, int32_t* __restrict__ counters)
{
    if (blockIdx.x == 0 && threadIdx.x == 0) counters[0] = 0;
    const int lane = threadIdx.x & 31;
    const int G = 1 << log2g;
    const int sub = lane & (G - 1);
    const int gpw = 32 >> log2g;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long base = warp * gpw; base < n_pix; base += nwarps * gpw) {
        const long long pix = base + (lane >> log2g);
        const bool valid = pix < n_pix;
        T a[PER];
        float s = 0.f;
        unsigned diff = 0;
#pragma unroll
        for (int k = 0; k < PER; ++k) {
            const int c = sub + k * G;
            if (valid && c < C) {
                a[k] = xt[pix * C + c];
                const T b = xp[pix * C + c];
                s += fabsf(to_f32(a[k]) - to_f32(b));
                if (sizeof(T) == 2) {
                    diff |= (unsigned)(*reinterpret_cast<const uint16_t*>(&a[k]) ^
                                       *reinterpret_cast<const uint16_t*>(&b));
                } else {
                    diff |= *reinterpret_cast<const uint32_t*>(&a[k]) ^ *reinterpret_cast<const uint32_t*>(&b);
                }
            }
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            if (off < G) {
                s += __shfl_xor_sync(0xffffffffu, s, off);
                diff |= __shfl_xor_sync(0xffffffffu, diff, off);
            }
        }
        if (valid) {
            if (diff || chg_prev[pix]) {
#pragma unroll
                for (int k = 0; k < PER; ++k) {
                    const int c = sub + k * G;
                    if (c < C) xn[pix * C + c] = a[k];
                }
            }
            if (sub == 0) {
                pix_l1[pix] = s;
                chg_cur[pix] = diff ? 1 : 0;
            }
        }
    }
}

// One warp per gate block.  The block's input footprint of per-pixel norms
// (FH x FW with FH = (b-1)*stride + k_h) is staged in shared memory with one
// round of coalesced loads; each lane then box-sums the supports of its
// output locations from shared memory.  When the footprint is too large for
// the staging area (stage == 0) the sums read global memory directly.
__global__ void __launch_bounds__(256) gate_block_kernel(
    const float* __restrict__ pix_l1, uint8_t* __restrict__ mask, int32_t* __restrict__ list,
    int32_t* __restrict__ counters, int n, int H, int W, int Ho, int Wo, int KH, int KW, int stride, int pad,
    int b, int nby, int nbx, float thr, int force, int stage)
{
    extern __shared__ float foot[];  // [8 warps][FH*FW] when staging
    __shared__ int flags[8];
    const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long nblocks = (long long)n * nby * nbx;
    const long long blk = (long long)blockIdx.x * 8 + wid;
    const int FH = (b - 1) * stride + KH, FW = (b - 1) * stride + KW;
    int open = 0;
    if (blk < nblocks) {
        if (force) {
            open = 1;
        } else {
            const int bx = (int)(blk % nbx);
            const long long rest = blk / nbx;
            const int by = (int)(rest % nby);
            const int nn = (int)(rest / nby);
            const float* P = pix_l1 + (size_t)nn * H * W;
            const int bh = min(b, Ho - by * b), bw = min(b, Wo - bx * b);
            const int fy0 = by * b * stride - pad, fx0 = bx * b * stride - pad;
            float* F = foot + wid * FH * FW;
            if (stage) {
                for (int q = lane; q < FH * FW; q += 32) {
                    const int yy = fy0 + q / FW, xx = fx0 + q % FW;
                    F[q] = (yy >= 0 && yy < H && xx >= 0 && xx < W) ? __ldg(P + (size_t)yy * W + xx) : 0.f;
                }
                __syncwarp();
            }
            float best = -1.f;
            for (int q = lane; q < bh * bw; q += 32) {
                const int i = q / bw, j = q % bw;  // within the block
                float S = 0.f;
                for (int kh = 0; kh < KH; ++kh)
                    for (int kw = 0; kw < KW; ++kw) {
                        const int fy = i * stride + kh, fx = j * stride + kw;
                        if (stage) {
                            S += F[fy * FW + fx];
                        } else {
                            const int yy = fy0 + fy, xx = fx0 + fx;
                            if (yy >= 0 && yy < H && xx >= 0 && xx < W) S += __ldg(P + (size_t)yy * W + xx);
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
        if (lane == 0 && bal) base = atomicAdd(&counters[0], __popc(bal));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (f) list[base + __popc(bal & ((1u << lane) - 1u))] = (int32_t)(blockIdx.x * 8 + lane);
    }
}

template <typename T>
cudaError_t launch_pixel_typed(const Layer& L, const void* x_t, const void* x_prev, void* x_next,
                               const uint8_t* chg_prev, uint8_t* chg_cur)
{
    const long long n_pix = (long long)L.p.n_streams * L.p.h * L.p.w;
    const int bytes = L.p.c_in * (int)sizeof(T);
    const bool vec = (bytes % 16 == 0) && ((uintptr_t)x_t % 16 == 0) && ((uintptr_t)x_prev % 16 == 0) &&
                     ((uintptr_t)x_next % 16 == 0);
    const int units = vec ? bytes / 16 : L.p.c_in;
    int log2g = 0;
    while ((1 << log2g) < units && log2g < 5) ++log2g;
    const int G = 1 << log2g;
    const int per = (units + G - 1) / G;
    const int gpw = 32 / G;
    long long warps_needed = (n_pix + gpw - 1) / gpw;
    long long blocks = (warps_needed + 7) / 8;
    const long long cap = (long long)L.num_sms * 8;
    const int grid = (int)(blocks < cap ? (blocks > 0 ? blocks : 1) : cap);
    if (vec) {
        const uint4* a = (const uint4*)x_t;
        const uint4* b = (const uint4*)x_prev;
        uint4* c = (uint4*)x_next;
        if (per == 1)
            gate_pixel_vec_kernel<T, 1, 1><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, log2g, L.counters);
        else if (per == 2)
            gate_pixel_vec_kernel<T, 2, 1><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, log2g, L.counters);
        else if (per <= 4)
            gate_pixel_vec_kernel<T, 4, 1><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, log2g, L.counters);
        else
            return cudaErrorInvalidValue;
    } else {
        const T* a = (const T*)x_t;
        const T* b = (const T*)x_prev;
        T* c = (T*)x_next;
        if (per == 1)
            gate_pixel_elem_kernel<T, 1><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, log2g, L.counters);
        else if (per == 2)
            gate_pixel_elem_kernel<T, 2><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, log2g, L.counters);
        else if (per <= 4)
            gate_pixel_elem_kernel<T, 4><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, log2g, L.counters);
        else if (per <= 8)
            gate_pixel_elem_kernel<T, 8><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, log2g, L.counters);
        else if (per <= 32)
            gate_pixel_elem_kernel<T, 32><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, log2g, L.counters);
        else
            return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace

// Largest channel count the gate kernels take (per pixel: 4 chunks of 16 B
// per lane on the vector path, 32 elements per lane on the element path).
int gate_max_channels(int dtype, bool vec)
{
    const int es = dtype == SKIPCONV_BF16 ? 2 : 4;
    return vec ? (32 * 4 * 16) / es : 32 * 32;
}

cudaError_t launch_gate_pixel(const Layer& L, const void* x_t, const void* x_prev, void* x_next,
                              const uint8_t* chg_prev, uint8_t* chg_cur)
{
    if (L.p.dtype == SKIPCONV_BF16)
        return launch_pixel_typed<__nv_bfloat16>(L, x_t, x_prev, x_next, chg_prev, chg_cur);
    return launch_pixel_typed<float>(L, x_t, x_prev, x_next, chg_prev, chg_cur);
}

cudaError_t launch_gate_block(const Layer& L, int force)
{
    const long long nblocks = (long long)L.p.n_streams * L.nby * L.nbx;
    const int grid = (int)((nblocks + 7) / 8);
    const int FH = (L.p.block - 1) * L.p.stride + L.p.k_h, FW = (L.p.block - 1) * L.p.stride + L.p.k_w;
    const size_t foot = (size_t)8 * FH * FW * sizeof(float);
    const int stage = foot <= 40 * 1024 ? 1 : 0;
    gate_block_kernel<<<grid, 256, stage ? foot : 0, L.stream>>>(
        L.pix_l1, L.mask, L.list, L.counters, L.p.n_streams, L.p.h, L.p.w, L.ho, L.wo, L.p.k_h, L.p.k_w,
        L.p.stride, L.p.pad, L.p.block, L.nby, L.nbx, L.gate_thr, force, stage);
    return cudaGetLastError();
}

}  // namespace sc
