// Gate kernels of the Skip-Conv step (two launches).
//
// Pass 1, per input pixel: the residual r_t = x_t - x_{t-1} (Eq. 2), its l1
// norm over all input channels (the channel part of the Input-Norm gate,
// Eq. 5, p = 1), and whether the pixel changed bit-wise.  The same pass
// commits x_t into the ping-pong buffer that becomes x_{t-1} at the next step,
// writing only pixels that changed at this step or the previous one (every
// other pixel of that buffer already holds x_t).
//
// Pass 2, per output block: the per-pixel norms summed over each output
// location's k_h x k_w receptive field (stride, zero padding) give the local
// support norm of Eq. 5; the block maximum (max-pooling of the gate,
// Sec. 3.2 on structured sparsity) is compared with the threshold and open
// blocks are appended to a compact list with one atomic per eight blocks.
//
// Pass 2 is a programmatic dependent launch of pass 1 (its launch latency
// hides behind pass 1's tail), and the convolution is one of pass 2.
// A single-launch form was tried: CTAs that publish a band of norms and let
// the last arriving band evaluate the block row spend about as long on the
// publication (fence, atomic, barrier) as on the streaming itself at these
// frame sizes, and were twice as slow.
#include "sc_internal.h"
#include "sc_ptx.cuh"

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

struct GateGeom {
    int n, H, W, Ho, Wo, KH, KW, stride, pad, b, nby, nbx;
};

// Max over the block's output locations of the support sum of per-pixel
// norms (one warp, returns the same value in every lane).  P is read from L2
// (other CTAs wrote it during this launch).
__device__ __forceinline__ float block_score(const GateGeom& g, const float* __restrict__ P, int nn, int by, int bx,
                                             int lane)
{
    const float* Pn = P + (size_t)nn * g.H * g.W;
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
                S += __ldcg(Pn + (size_t)yy * g.W + xx);
            }
        }
        best = fmaxf(best, S);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, off));
    return best;
}

// Vector path, pass 1 of 2: every warp of a grid-stride grid takes groups of
// pixels (G lanes per pixel, PER 16-byte chunks per lane); the change flag of
// the previous step is loaded together with the frames.  The last thing each
// CTA does is let the block-gate pass start (programmatic dependent launch).
template <typename T, int PER>
__global__ void __launch_bounds__(256) gate_pixel_vec_kernel(
    const uint4* __restrict__ xt, const uint4* __restrict__ xp, uint4* __restrict__ xn,
    const uint8_t* __restrict__ chg_prev, uint8_t* __restrict__ chg_cur, float* __restrict__ pix_l1,
    long long n_pix, int cpp, int log2g, int32_t* __restrict__ count_cur, int32_t* __restrict__ count_next)
{
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        *count_cur = 0;   // this step's active-block count (filled by the block-gate pass)
        *count_next = 0;
    }
    const int lane = threadIdx.x & 31;
    const int G = 1 << log2g;
    const int sub = lane & (G - 1);
    const int gpw = 32 >> log2g;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long base = warp * gpw; base < n_pix; base += nwarps * gpw) {
        const long long pix = base + (lane >> log2g);
        const bool valid = pix < n_pix;
        uint4 a[PER], b[PER];
        const uint8_t cprev = valid ? __ldg(chg_prev + pix) : (uint8_t)0;
#pragma unroll
        for (int k = 0; k < PER; ++k) {
            const int c = sub + k * G;
            if (valid && c < cpp) {
                a[k] = __ldg(xt + pix * cpp + c);
                b[k] = __ldg(xp + pix * cpp + c);
            } else {
                a[k] = make_uint4(0, 0, 0, 0);
                b[k] = make_uint4(0, 0, 0, 0);
            }
        }
        float s = 0.f;
        unsigned diff = 0;
#pragma unroll
        for (int k = 0; k < PER; ++k) {
            s += l1_diff(a[k], b[k], (T*)nullptr);
            diff |= bits_differ(a[k], b[k]);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
            if (off < G) {
                s += __shfl_xor_sync(0xffffffffu, s, off);
                diff |= __shfl_xor_sync(0xffffffffu, diff, off);
            }
        }
        if (valid) {
            if (diff || cprev) {
#pragma unroll
                for (int k = 0; k < PER; ++k) {
                    const int c = sub + k * G;
                    if (c < cpp) xn[pix * cpp + c] = a[k];
                }
            }
            if (sub == 0) {
                pix_l1[pix] = s;
                chg_cur[pix] = diff ? 1 : 0;
            }
        }
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Element path for channel counts whose pixel is not a multiple of 16 bytes.
template <typename T, int PER>
__global__ void __launch_bounds__(256) gate_pixel_elem_kernel(
    const T* __restrict__ xt, const T* __restrict__ xp, T* __restrict__ xn,
    const uint8_t* __restrict__ chg_prev, uint8_t* __restrict__ chg_cur, float* __restrict__ pix_l1,
    long long n_pix, int C, int log2g, int32_t* __restrict__ count_cur, int32_t* __restrict__ count_next)
{
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        *count_cur = 0;
        *count_next = 0;
    }
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
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// One warp per gate block (two-launch form).
// Pass 2: one warp per gate block.  Launched as a programmatic dependent of
// pass 1: it waits for pass 1's results before reading them, and lets the
// convolution after it start its own prologue right away.  When the block's
// footprint of norms fits (stage), it is staged in shared memory with one
// round of loads.
__global__ void __launch_bounds__(256) gate_block_kernel(const float* __restrict__ pix_l1, uint8_t* __restrict__ mask,
                                                         int32_t* __restrict__ list, int32_t* __restrict__ count_cur,
                                                         GateGeom g, float thr, int force, int stage)
{
    extern __shared__ float foot[];  // [8 warps][FH * FW]
    __shared__ int flags[8];
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
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
            if (stage) {
                // block footprint (FH x FW) into this warp's slice of shared memory
                const int FH = (g.b - 1) * g.stride + g.KH, FW = (g.b - 1) * g.stride + g.KW;
                float* F = foot + wid * FH * FW;
                const float* Pn = pix_l1 + (size_t)nn * g.H * g.W;
                const int fy0 = by * g.b * g.stride - g.pad, fx0 = bx * g.b * g.stride - g.pad;
                for (int q = lane; q < FH * FW; q += 32) {
                    const int yy = fy0 + q / FW, xx = fx0 + q % FW;
                    F[q] = (yy >= 0 && yy < g.H && xx >= 0 && xx < g.W) ? __ldcg(Pn + (size_t)yy * g.W + xx) : 0.f;
                }
                __syncwarp();
                const int bh = min(g.b, g.Ho - by * g.b), bw = min(g.b, g.Wo - bx * g.b);
                float best = -1.f;
                for (int q = lane; q < bh * bw; q += 32) {
                    const int i = q / bw, j = q - (q / bw) * bw;
                    float S = 0.f;
                    for (int kh = 0; kh < g.KH; ++kh)
                        for (int kw = 0; kw < g.KW; ++kw) S += F[(i * g.stride + kh) * FW + j * g.stride + kw];
                    best = fmaxf(best, S);
                }
#pragma unroll
                for (int off = 16; off > 0; off >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, off));
                open = best > thr ? 1 : 0;
            } else {
                open = block_score(g, pix_l1, nn, by, bx, lane) > thr ? 1 : 0;
            }
        }
        if (lane == 0) mask[blk] = (uint8_t)open;
    }
    if (lane == 0) flags[wid] = open;
    __syncthreads();
    if (wid == 0) {
        const int f = lane < 8 ? flags[lane] : 0;
        const unsigned bal = __ballot_sync(0xffffffffu, f);
        int base = 0;
        if (lane == 0 && bal) base = atomicAdd(count_cur, __popc(bal));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (f) list[base + __popc(bal & ((1u << lane) - 1u))] = (int32_t)(blockIdx.x * 8 + lane);
    }
}

// Gumbel gate (Eq. 8 at inference), pass 1 of 2: one warp per input pixel.
// The gate function f(r; phi) is a convolution of r with one output channel
// and the layer's kernel; this pass forms, for each of the k_h*k_w taps t,
// the pixel's partial product d_t = sum_c phi[t][c] r[c] (phi staged in shared
// memory as [tap][channel]), plus the change flag and the state commit of the
// norm pass.  Pass 2 sums the taps' partial products over each output
// location's receptive field.
constexpr int GUMBEL_MAX_TAPS = 9;

template <typename T>
__global__ void __launch_bounds__(256) gate_pixel_gumbel_kernel(
    const T* __restrict__ xt, const T* __restrict__ xp, T* __restrict__ xn, const uint8_t* __restrict__ chg_prev,
    uint8_t* __restrict__ chg_cur, const float* __restrict__ phi, float* __restrict__ taps_out, long long n_pix, int C,
    int taps, int32_t* __restrict__ count_cur, int32_t* __restrict__ count_next)
{
    extern __shared__ float sphi[];  // [taps][C]
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        *count_cur = 0;
        *count_next = 0;
    }
    for (int i = threadIdx.x; i < taps * C; i += blockDim.x) sphi[i] = phi[i];
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long pix = warp; pix < n_pix; pix += nwarps) {
        float acc[GUMBEL_MAX_TAPS];
#pragma unroll
        for (int t = 0; t < GUMBEL_MAX_TAPS; ++t) acc[t] = 0.f;
        unsigned diff = 0;
        for (int c = lane; c < C; c += 32) {
            const T a = xt[pix * C + c], b = xp[pix * C + c];
            const float r = to_f32(a) - to_f32(b);
            if (sizeof(T) == 2)
                diff |= (unsigned)(*reinterpret_cast<const uint16_t*>(&a) ^ *reinterpret_cast<const uint16_t*>(&b));
            else
                diff |= *reinterpret_cast<const uint32_t*>(&a) ^ *reinterpret_cast<const uint32_t*>(&b);
#pragma unroll
            for (int t = 0; t < GUMBEL_MAX_TAPS; ++t)
                if (t < taps) acc[t] = fmaf(sphi[t * C + c], r, acc[t]);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) {
#pragma unroll
            for (int t = 0; t < GUMBEL_MAX_TAPS; ++t) acc[t] += __shfl_xor_sync(0xffffffffu, acc[t], off);
            diff |= __shfl_xor_sync(0xffffffffu, diff, off);
        }
        if (diff || chg_prev[pix])
            for (int c = lane; c < C; c += 32) xn[pix * C + c] = xt[pix * C + c];
        if (lane == 0) {
#pragma unroll
            for (int t = 0; t < GUMBEL_MAX_TAPS; ++t)
                if (t < taps) taps_out[pix * taps + t] = acc[t];
            chg_cur[pix] = diff ? 1 : 0;
        }
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// The same pass for pixels of 16-byte vectors: G = 2^LOG2G lanes per pixel
// (8 to 32), each with one 16-byte vector of both frames, 32 / G pixels per
// warp.  A lane forms its channels' share of all taps (phi from shared
// memory, four floats per load); the pixel's G shares of taps 0-7 are summed
// by a transposed butterfly (three halving exchanges leave one tap's partial
// sum in each lane, then plain steps) and tap 8 by a plain one, so every tap
// costs a fraction of a butterfly of its own.
__device__ __forceinline__ void unpack8(const uint4& v, float (&f)[8], const __nv_bfloat16*)
{
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 t = __bfloat1622float2(h[k]);
        f[2 * k] = t.x;
        f[2 * k + 1] = t.y;
    }
}
__device__ __forceinline__ void unpack8(const uint4& v, float (&f)[8], const float*)
{
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y); f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
    f[4] = f[5] = f[6] = f[7] = 0.f;
}

template <typename T, int LOG2G>
__global__ void __launch_bounds__(256) gate_pixel_gumbel_vec_kernel(
    const T* __restrict__ xt, const T* __restrict__ xp, T* __restrict__ xn, const uint8_t* __restrict__ chg_prev,
    uint8_t* __restrict__ chg_cur, const float* __restrict__ phi, float* __restrict__ taps_out, long long n_pix, int C,
    int taps, int32_t* __restrict__ count_cur, int32_t* __restrict__ count_next)
{
    constexpr int G = 1 << LOG2G, PPW = 32 / G, VX = 16 / (int)sizeof(T);
    constexpr int PL = 2;   // pixels per lane and pass: their loads go out together, phi is read once for both
    extern __shared__ float sphi[];  // [GUMBEL_MAX_TAPS][C], taps past `taps` zero
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        *count_cur = 0;
        *count_next = 0;
    }
    for (int i = threadIdx.x; i < GUMBEL_MAX_TAPS * C; i += blockDim.x) sphi[i] = i < taps * C ? phi[i] : 0.f;
    __syncthreads();
    const int lane = threadIdx.x & 31, sub = lane & (G - 1), prow = lane >> LOG2G;
    const int units = C / VX;
    const bool lane_on = sub < units;
    const int c0 = sub * VX;
    // the tap whose sum this lane holds after the halving exchanges
    const int my_tap = (((sub >> (LOG2G - 1)) & 1) << 2) | (((sub >> (LOG2G - 2)) & 1) << 1) | ((sub >> (LOG2G - 3)) & 1);
    const bool writer = (sub & ((G >> 3) - 1)) == 0;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long long nwarps = ((long long)gridDim.x * blockDim.x) >> 5;
    for (long long p0 = warp * PPW * PL; p0 < n_pix; p0 += nwarps * PPW * PL) {
        long long pix[PL];
        bool on[PL];
        uint4 av[PL], bv[PL];
#pragma unroll
        for (int u = 0; u < PL; ++u) {
            pix[u] = p0 + u * PPW + prow;
            on[u] = lane_on && pix[u] < n_pix;
            av[u] = make_uint4(0, 0, 0, 0);
            bv[u] = av[u];
            if (on[u]) {
                av[u] = reinterpret_cast<const uint4*>(xt + pix[u] * C)[sub];
                bv[u] = reinterpret_cast<const uint4*>(xp + pix[u] * C)[sub];
            }
        }
        float r[PL][8], acc[PL][GUMBEL_MAX_TAPS];
        unsigned d[PL];
#pragma unroll
        for (int u = 0; u < PL; ++u) {
            d[u] = (av[u].x ^ bv[u].x) | (av[u].y ^ bv[u].y) | (av[u].z ^ bv[u].z) | (av[u].w ^ bv[u].w);
            float fa[8], fb[8];
            unpack8(av[u], fa, (const T*)nullptr);
            unpack8(bv[u], fb, (const T*)nullptr);
#pragma unroll
            for (int j = 0; j < 8; ++j) r[u][j] = fa[j] - fb[j];
#pragma unroll
            for (int t = 0; t < GUMBEL_MAX_TAPS; ++t) acc[u][t] = 0.f;
        }
        if (lane_on) {
#pragma unroll
            for (int t = 0; t < GUMBEL_MAX_TAPS; ++t) {
                const float4 w0 = *reinterpret_cast<const float4*>(sphi + t * C + c0);
                const float4 w1 = VX == 8 ? *reinterpret_cast<const float4*>(sphi + t * C + c0 + 4)
                                          : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int u = 0; u < PL; ++u) {
                    float a = 0.f;
                    a = fmaf(w0.x, r[u][0], a);
                    a = fmaf(w0.y, r[u][1], a);
                    a = fmaf(w0.z, r[u][2], a);
                    a = fmaf(w0.w, r[u][3], a);
                    if (VX == 8) {
                        a = fmaf(w1.x, r[u][4], a);
                        a = fmaf(w1.y, r[u][5], a);
                        a = fmaf(w1.z, r[u][6], a);
                        a = fmaf(w1.w, r[u][7], a);
                    }
                    acc[u][t] = a;
                }
            }
        }
#pragma unroll
        for (int u = 0; u < PL; ++u) {
            // taps 0-7: transposed butterfly over the pixel's G lanes
            float t4[4], t2[2], t1;
            {
                const bool h = (sub >> (LOG2G - 1)) & 1;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float send = h ? acc[u][q] : acc[u][q + 4], keep = h ? acc[u][q + 4] : acc[u][q];
                    t4[q] = keep + __shfl_xor_sync(0xffffffffu, send, G >> 1);
                }
            }
            {
                const bool h = (sub >> (LOG2G - 2)) & 1;
#pragma unroll
                for (int q = 0; q < 2; ++q) {
                    const float send = h ? t4[q] : t4[q + 2], keep = h ? t4[q + 2] : t4[q];
                    t2[q] = keep + __shfl_xor_sync(0xffffffffu, send, G >> 2);
                }
            }
            {
                const bool h = (sub >> (LOG2G - 3)) & 1;
                const float send = h ? t2[0] : t2[1], keep = h ? t2[1] : t2[0];
                t1 = keep + __shfl_xor_sync(0xffffffffu, send, G >> 3);
            }
#pragma unroll
            for (int off = G >> 4; off > 0; off >>= 1) t1 += __shfl_xor_sync(0xffffffffu, t1, off);
            // tap 8 and the change bits: plain butterflies within the pixel's lanes
            float a8 = acc[u][8];
            unsigned du = d[u];
#pragma unroll
            for (int off = G >> 1; off > 0; off >>= 1) {
                a8 += __shfl_xor_sync(0xffffffffu, a8, off);
                du |= __shfl_xor_sync(0xffffffffu, du, off);
            }
            if (pix[u] < n_pix) {
                const bool changed = du != 0;
                if (on[u] && (changed || chg_prev[pix[u]])) reinterpret_cast<uint4*>(xn + pix[u] * C)[sub] = av[u];
                if (writer && my_tap < taps) taps_out[pix[u] * taps + my_tap] = t1;
                if (sub == 0) {
                    if (taps > 8) taps_out[pix[u] * taps + 8] = a8;
                    chg_cur[pix[u]] = changed ? 1 : 0;
                }
            }
        }
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// The same pass for 512-byte pixels (32 lanes x 16 bytes: 256 bf16 or 128
// fp32 channels), streamed: a persistent grid of one CTA per SM, each warp
// refilling its own GS_NSLOT shared-memory slots by bulk copies with chunks of
// GS_ROWS pixels of both frames, so the bytes in flight do not occupy registers.  A
// warp takes a whole chunk at once: phi is read once per chunk and shared by
// its GS_ROWS pixels, and the GS_ROWS x 9 tap sums are reduced over the 32
// lanes by a transposed butterfly (halving exchanges leave one pixel's 9 sums in
// each lane, then plain steps).  Waits are bounded; one that runs out
// records a timeout in the error word.
constexpr int GS_WARPS = 8;
constexpr int GS_ROWS = 8;                       // pixels per chunk

// Packed pairs of fp32 values (one 64-bit register) and the sm_100-family
// paired arithmetic on them: each lane of a pair is the IEEE fp32 operation
// with round to nearest, exactly what the scalar instruction computes, in
// half the instructions.
__device__ __forceinline__ unsigned long long f2pack(float lo, float hi)
{
    unsigned long long r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void f2unpack(unsigned long long v, float& lo, float& hi)
{
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ unsigned long long f2sub(unsigned long long a, unsigned long long b)
{
    unsigned long long d;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ unsigned long long f2mul(unsigned long long a, unsigned long long b)
{
    unsigned long long d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ unsigned long long f2fma(unsigned long long a, unsigned long long b, unsigned long long c)
{
    unsigned long long d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}
constexpr int GS_HALF = GS_ROWS * 512;           // one frame's chunk
constexpr int GS_SLOT = 2 * GS_HALF;
constexpr int GS_NSLOT = 2;                      // chunks in flight per warp
constexpr uint64_t GS_WAIT_NS = 1000000000ull;

size_t gumbel_stream_smem_bytes() { return 128 + (size_t)GUMBEL_MAX_TAPS * 256 * 4 + (size_t)GS_WARPS * GS_NSLOT * GS_SLOT; }

template <typename T>
__global__ void __launch_bounds__(GS_WARPS * 32, 1) gate_pixel_gumbel_stream_kernel(
    const T* __restrict__ xt, const T* __restrict__ xp, T* __restrict__ xn, const uint8_t* __restrict__ chg_prev,
    uint8_t* __restrict__ chg_cur, const float* __restrict__ phi, float* __restrict__ taps_out, long long n_pix,
    int taps, int32_t* __restrict__ count_cur, int32_t* __restrict__ count_next, int* __restrict__ err)
{
    constexpr int VX = 16 / (int)sizeof(T), C = 32 * VX;
    extern __shared__ uint8_t gsm_raw[];
    uint8_t* gsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(gsm_raw) + 127) & ~(uintptr_t)127);
    float* sphi = reinterpret_cast<float*>(gsm);                       // [GUMBEL_MAX_TAPS][C]
    uint8_t* ring = gsm + GUMBEL_MAX_TAPS * 256 * 4;                  // [warp][slot][x_t | x_{t-1}]
    __shared__ __align__(8) uint64_t full[GS_WARPS][GS_NSLOT];
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        *count_cur = 0;
        *count_next = 0;
    }
    if (threadIdx.x == 0) {
        for (int w = 0; w < GS_WARPS; ++w)
            for (int q = 0; q < GS_NSLOT; ++q) ptx::mbar_init(ptx::smem_u32(&full[w][q]), 1);
        ptx::fence_mbar_init();
    }
    for (int i = threadIdx.x; i < GUMBEL_MAX_TAPS * C; i += blockDim.x) sphi[i] = i < taps * C ? phi[i] : 0.f;
    __syncthreads();
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const long long nch = (n_pix + GS_ROWS - 1) / GS_ROWS;
    const long long k0 = (long long)blockIdx.x * GS_WARPS + wid, ks = (long long)gridDim.x * GS_WARPS;
    uint8_t* slots = ring + wid * GS_NSLOT * GS_SLOT;
    auto issue = [&](long long k, int q) {
        const long long p0 = k * GS_ROWS;
        const int np = (int)min((long long)GS_ROWS, n_pix - p0);
        const uint32_t bytes = (uint32_t)(np * 512);
        const uint32_t bar = ptx::smem_u32(&full[wid][q]);
        ptx::mbar_arrive_expect_tx(bar, 2 * bytes);
        ptx::bulk_load(ptx::smem_u32(slots + q * GS_SLOT), xt + p0 * C, bytes, bar);
        ptx::bulk_load(ptx::smem_u32(slots + q * GS_SLOT + GS_HALF), xp + p0 * C, bytes, bar);
    };
    if (lane == 0)
        for (int i = 0; i < GS_NSLOT; ++i)
            if (k0 + i * ks < nch) issue(k0 + i * ks, i);
    uint32_t phases = 0;
    int q = 0;
    for (long long k = k0; k < nch; k += ks) {
        const long long p0 = k * GS_ROWS;
        const int np = (int)min((long long)GS_ROWS, n_pix - p0);
        const uint32_t cprev = lane < np ? chg_prev[p0 + lane] : 0u;   // lanes below np: the chunk's previous flags
        const uint32_t bar = ptx::smem_u32(&full[wid][q]);
        const bool ok = __all_sync(0xffffffffu, ptx::mbar_wait(bar, (phases >> q) & 1u, nullptr, err, GS_WAIT_NS)) != 0;
        if (!ok) {
            // the copies in flight may still land: wait for them (bounded) before the CTA can exit
            if (lane == 0)
                for (int i = 0; i < GS_NSLOT; ++i) {
                    const int qi = (q + i) % GS_NSLOT;
                    if (k + i * ks < nch)
                        ptx::mbar_wait(ptx::smem_u32(&full[wid][qi]), (phases >> qi) & 1u, nullptr, nullptr, GS_WAIT_NS);
                }
            return;
        }
        const uint4* sx = reinterpret_cast<const uint4*>(slots + q * GS_SLOT);
        const uint4* sp = reinterpret_cast<const uint4*>(slots + q * GS_SLOT + GS_HALF);
        // residuals of rows 2i and 2i+1 packed in pairs: r2[i][j] = (r[2i][j], r[2i+1][j])
        unsigned long long r2[GS_ROWS / 2][8];
        float fa_even[8], fb_even[8];
        uint32_t chg_rows = 0;   // bit row: the pixel changed
#pragma unroll
        for (int row = 0; row < GS_ROWS; ++row) {
            uint4 av = make_uint4(0, 0, 0, 0), bv = av;
            if (row < np) {
                av = sx[row * 32 + lane];
                bv = sp[row * 32 + lane];
            }
            const bool dif = ((av.x ^ bv.x) | (av.y ^ bv.y) | (av.z ^ bv.z) | (av.w ^ bv.w)) != 0u;
            const bool changed = __any_sync(0xffffffffu, dif);
            chg_rows |= (changed ? 1u : 0u) << row;
            const uint32_t cp = __shfl_sync(0xffffffffu, cprev, row);
            if (row < np && (changed || cp != 0u)) reinterpret_cast<uint4*>(xn + (p0 + row) * C)[lane] = av;
            float fa[8], fb[8];
            unpack8(av, fa, (const T*)nullptr);
            unpack8(bv, fb, (const T*)nullptr);
            if ((row & 1) == 0) {
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    fa_even[j] = fa[j];
                    fb_even[j] = fb[j];
                }
            } else {
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    r2[row / 2][j] = f2sub(f2pack(fa_even[j], fa[j]), f2pack(fb_even[j], fb[j]));
            }
        }
        __syncwarp();
        if (lane == 0 && k + GS_NSLOT * ks < nch) {
            ptx::fence_proxy_async_smem();   // the slot's reads before the copy that overwrites it
            issue(k + GS_NSLOT * ks, q);
        }
        phases ^= 1u << q;
        q = q + 1 == GS_NSLOT ? 0 : q + 1;
        // the chunk's tap products: v[row * 9 + t] = sum over this lane's channels of phi[t][c] r[c]
        // (the products and sums of each row are the scalar sequence mul, fma, fma, ...: two rows per instruction)
        float v[GS_ROWS * GUMBEL_MAX_TAPS];
#pragma unroll
        for (int t = 0; t < GUMBEL_MAX_TAPS; ++t) {
            const float4 w0 = *reinterpret_cast<const float4*>(sphi + t * C + lane * VX);
            const float4 w1 = VX == 8 ? *reinterpret_cast<const float4*>(sphi + t * C + lane * VX + 4)
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
            const unsigned long long p0 = f2pack(w0.x, w0.x), p1 = f2pack(w0.y, w0.y), p2 = f2pack(w0.z, w0.z),
                                     p3 = f2pack(w0.w, w0.w), p4 = f2pack(w1.x, w1.x), p5 = f2pack(w1.y, w1.y),
                                     p6 = f2pack(w1.z, w1.z), p7 = f2pack(w1.w, w1.w);
#pragma unroll
            for (int i = 0; i < GS_ROWS / 2; ++i) {
                unsigned long long a = f2mul(p0, r2[i][0]);
                a = f2fma(p1, r2[i][1], a);
                a = f2fma(p2, r2[i][2], a);
                a = f2fma(p3, r2[i][3], a);
                if (VX == 8) {
                    a = f2fma(p4, r2[i][4], a);
                    a = f2fma(p5, r2[i][5], a);
                    a = f2fma(p6, r2[i][6], a);
                    a = f2fma(p7, r2[i][7], a);
                }
                f2unpack(a, v[(2 * i) * GUMBEL_MAX_TAPS + t], v[(2 * i + 1) * GUMBEL_MAX_TAPS + t]);
            }
        }
        // transposed butterfly: each halving exchange keeps half of the rows, until one row's 9 sums are
        // left in each lane; then plain steps over the remaining lanes of that row
        static_assert(GS_ROWS == 4 || GS_ROWS == 8, "rows per chunk");
        constexpr int N1 = GS_ROWS * GUMBEL_MAX_TAPS / 2, N2 = N1 / 2;
        float v1[N1], v2[N2];
        {
            const bool h = (lane >> 4) & 1;
#pragma unroll
            for (int i = 0; i < N1; ++i) {
                const float send = h ? v[i] : v[i + N1], keep = h ? v[i + N1] : v[i];
                v1[i] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
            }
        }
        {
            const bool h = (lane >> 3) & 1;
#pragma unroll
            for (int i = 0; i < N2; ++i) {
                const float send = h ? v1[i] : v1[i + N2], keep = h ? v1[i + N2] : v1[i];
                v2[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
            }
        }
        float v3[GUMBEL_MAX_TAPS];
        int row;
        if (GS_ROWS == 8) {
            const bool h = (lane >> 2) & 1;
#pragma unroll
            for (int i = 0; i < GUMBEL_MAX_TAPS; ++i) {
                const float send = h ? v2[i] : v2[(i + GUMBEL_MAX_TAPS) % N2], keep = h ? v2[(i + GUMBEL_MAX_TAPS) % N2] : v2[i];
                v3[i] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
            }
#pragma unroll
            for (int i = 0; i < GUMBEL_MAX_TAPS; ++i) {
                v3[i] += __shfl_xor_sync(0xffffffffu, v3[i], 2);
                v3[i] += __shfl_xor_sync(0xffffffffu, v3[i], 1);
            }
            row = (((lane >> 4) & 1) << 2) | (((lane >> 3) & 1) << 1) | ((lane >> 2) & 1);
        } else {
#pragma unroll
            for (int i = 0; i < GUMBEL_MAX_TAPS; ++i) {
                v3[i] = v2[i % N2];
                v3[i] += __shfl_xor_sync(0xffffffffu, v3[i], 4);
                v3[i] += __shfl_xor_sync(0xffffffffu, v3[i], 2);
                v3[i] += __shfl_xor_sync(0xffffffffu, v3[i], 1);
            }
            row = (((lane >> 4) & 1) << 1) | ((lane >> 3) & 1);
        }
        // lane holds the 9 sums of pixel `row`; one lane per row writes them
        if ((lane & (32 / GS_ROWS - 1)) == 0 && row < np) {
#pragma unroll
            for (int t = 0; t < GUMBEL_MAX_TAPS; ++t)
                if (t < taps) taps_out[(p0 + row) * taps + t] = v3[t];
        }
        if (lane < np) chg_cur[p0 + lane] = (chg_rows >> lane) & 1u;
    }
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Gumbel gate, pass 2 of 2: one warp per gate block.  f at an output location
// is phi_bias plus the partial products of the taps over its receptive field
// (zero padding: out-of-frame taps add nothing); the block opens when its
// largest f exceeds the threshold (eps; eps = 0 is round(sigmoid(f)) = 1).
__global__ void __launch_bounds__(256) gate_block_gumbel_kernel(const float* __restrict__ taps_in,
                                                                uint8_t* __restrict__ mask, int32_t* __restrict__ list,
                                                                int32_t* __restrict__ count_cur, GateGeom g,
                                                                float thr, float phi_bias, int force)
{
    __shared__ int flags[8];
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int wid = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int taps = g.KH * g.KW;
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
            const float* Tn = taps_in + (size_t)nn * g.H * g.W * taps;
            const int bh = min(g.b, g.Ho - by * g.b), bw = min(g.b, g.Wo - bx * g.b);
            const int fy0 = by * g.b * g.stride - g.pad, fx0 = bx * g.b * g.stride - g.pad;
            float best = -INFINITY;
            if (g.KH == 3 && g.KW == 3 && bh * bw <= 64) {
                // 3x3: a lane's (up to) two outputs issue all 18 loads before summing (out-of-frame taps add
                // 0, which leaves the sum as skipping them would)
                float t[2][9];
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int q = lane + 32 * u;
                    const bool on = q < bh * bw;
                    const int i = on ? q / bw : 0, j = on ? q - (q / bw) * bw : 0;
#pragma unroll
                    for (int kk = 0; kk < 9; ++kk) {
                        const int yy = fy0 + i * g.stride + kk / 3, xx = fx0 + j * g.stride + kk % 3;
                        const bool in = on && yy >= 0 && yy < g.H && xx >= 0 && xx < g.W;
                        t[u][kk] = in ? __ldcg(Tn + ((size_t)yy * g.W + xx) * 9 + kk) : 0.f;
                    }
                }
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    if (lane + 32 * u >= bh * bw) continue;
                    float f = phi_bias;
#pragma unroll
                    for (int kk = 0; kk < 9; ++kk) f += t[u][kk];
                    best = fmaxf(best, f);
                }
            } else {
                for (int q = lane; q < bh * bw; q += 32) {
                    const int i = q / bw, j = q - (q / bw) * bw;
                    float f = phi_bias;
                    for (int kh = 0; kh < g.KH; ++kh) {
                        const int yy = fy0 + i * g.stride + kh;
                        if (yy < 0 || yy >= g.H) continue;
                        for (int kw = 0; kw < g.KW; ++kw) {
                            const int xx = fx0 + j * g.stride + kw;
                            if (xx < 0 || xx >= g.W) continue;
                            f += __ldcg(Tn + ((size_t)yy * g.W + xx) * taps + kh * g.KW + kw);
                        }
                    }
                    best = fmaxf(best, f);
                }
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
        if (lane == 0 && bal) base = atomicAdd(count_cur, __popc(bal));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (f) list[base + __popc(bal & ((1u << lane) - 1u))] = (int32_t)(blockIdx.x * 8 + lane);
    }
}

GateGeom geom_of(const Layer& L)
{
    GateGeom g;
    g.n = L.p.n_streams;
    g.H = L.p.h;
    g.W = L.p.w;
    g.Ho = L.ho;
    g.Wo = L.wo;
    g.KH = L.p.k_h;
    g.KW = L.p.k_w;
    g.stride = L.p.stride;
    g.pad = L.p.pad;
    g.b = L.p.block;
    g.nby = L.nby;
    g.nbx = L.nbx;
    return g;
}

template <typename T>
cudaError_t launch_typed(const Layer& L, const void* x_t, const void* x_prev, void* x_next, const uint8_t* chg_prev,
                         uint8_t* chg_cur, int force)
{
    int32_t* cnt_cur = step_count(L);
    int32_t* cnt_next = next_count(L);
    const int bytes = L.p.c_in * (int)sizeof(T);
    const bool vec = (bytes % 16 == 0) && ((uintptr_t)x_t % 16 == 0) && ((uintptr_t)x_prev % 16 == 0) &&
                     ((uintptr_t)x_next % 16 == 0);
    const int units = vec ? bytes / 16 : L.p.c_in;
    int log2g = 0;
    while ((1 << log2g) < units && log2g < 5) ++log2g;
    const int G = 1 << log2g;
    const int per = (units + G - 1) / G;
    const GateGeom g = geom_of(L);
    const long long n_pix = (long long)L.p.n_streams * L.p.h * L.p.w;
    const int gpw = 32 / G;
    const long long warps_needed = (n_pix + gpw - 1) / gpw;
    const long long blocks = (warps_needed + 7) / 8;
    const long long cap = (long long)L.num_sms * 8;
    const int grid = (int)(blocks < cap ? (blocks > 0 ? blocks : 1) : cap);
    if (vec) {
        const uint4* a = (const uint4*)x_t;
        const uint4* b = (const uint4*)x_prev;
        uint4* c = (uint4*)x_next;
#define SC_VEC(PER_)                                                                                             \
    gate_pixel_vec_kernel<T, PER_><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, \
                                                               log2g, cnt_cur, cnt_next)
        if (per == 1) SC_VEC(1);
        else if (per == 2) SC_VEC(2);
        else if (per <= 4) SC_VEC(4);
        else return cudaErrorInvalidValue;
#undef SC_VEC
    } else {
    const T* a = (const T*)x_t;
    const T* b = (const T*)x_prev;
    T* c = (T*)x_next;
#define SC_ELEM(PER_)                                                                                              \
    gate_pixel_elem_kernel<T, PER_><<<grid, 256, 0, L.stream>>>(a, b, c, chg_prev, chg_cur, L.pix_l1, n_pix, units, \
                                                                log2g, cnt_cur, cnt_next)
    if (per == 1) SC_ELEM(1);
    else if (per == 2) SC_ELEM(2);
    else if (per <= 4) SC_ELEM(4);
    else if (per <= 8) SC_ELEM(8);
    else if (per <= 32) SC_ELEM(32);
    else return cudaErrorInvalidValue;
#undef SC_ELEM
    }
    (void)force;
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gate_blocks(const Layer& L, int force)
{
    int32_t* cnt_cur = step_count(L);
    const GateGeom g = geom_of(L);
    const long long nblocks = (long long)L.p.n_streams * L.nby * L.nbx;
    const int FH = (L.p.block - 1) * L.p.stride + L.p.k_h, FW = (L.p.block - 1) * L.p.stride + L.p.k_w;
    const size_t foot = (size_t)8 * FH * FW * sizeof(float);
    const int stage = foot <= 40 * 1024 ? 1 : 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((nblocks + 7) / 8));
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = stage ? foot : 0;
    cfg.stream = L.stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, gate_block_kernel, (const float*)L.pix_l1, L.mask, L.list, cnt_cur, g,
                              L.gate_thr, force, stage);
}

// Largest channel count the gate kernels take (per pixel: 4 chunks of 16 B
// per lane on the vector path, 32 elements per lane on the element path).
int gate_max_channels(int dtype, bool vec)
{
    const int es = dtype == SKIPCONV_BF16 ? 2 : 4;
    return vec ? (32 * 4 * 16) / es : 32 * 32;
}

// lanes per pixel of the vector form (2^k, 8 to 32), or 0 when the pixel is not whole 16-byte vectors
static int gumbel_vec_log2g(const Layer& L)
{
    if ((L.p.c_in * L.esize) % 16 != 0 || L.p.k_h * L.p.k_w > GUMBEL_MAX_TAPS) return 0;
    const int units = L.p.c_in * L.esize / 16;
    if (units > 32) return 0;
    int lg = 3;
    while ((1 << lg) < units) ++lg;
    return lg;
}

// the streamed form: 512-byte pixels and at most GUMBEL_MAX_TAPS taps
static bool gumbel_streamed(const Layer& L)
{
    return L.p.c_in * L.esize == 512 && L.p.k_h * L.p.k_w <= GUMBEL_MAX_TAPS;
}

cudaError_t gumbel_prepare(const Layer& L)
{
    if (!gumbel_streamed(L)) return cudaSuccess;
    return L.p.dtype == SKIPCONV_BF16
               ? ensure_dynamic_smem((const void*)gate_pixel_gumbel_stream_kernel<__nv_bfloat16>, gumbel_stream_smem_bytes())
               : ensure_dynamic_smem((const void*)gate_pixel_gumbel_stream_kernel<float>, gumbel_stream_smem_bytes());
}

// phi in shared memory: [taps][c_in]; the vector form pads it to GUMBEL_MAX_TAPS taps (c_in <= 256 there)
size_t gumbel_smem_bytes(const Layer& L)
{
    const int taps = gumbel_vec_log2g(L) ? GUMBEL_MAX_TAPS : L.p.k_h * L.p.k_w;
    return (size_t)taps * L.p.c_in * sizeof(float);
}

cudaError_t launch_gate_pixels_gumbel(const Layer& L, const void* x_t, const void* x_prev, void* x_next,
                                      const uint8_t* chg_prev, uint8_t* chg_cur)
{
    const long long n_pix = (long long)L.p.n_streams * L.p.h * L.p.w;
    const long long blocks = (n_pix + 7) / 8;
    const long long cap = (long long)L.num_sms * 8;
    const int grid = (int)(blocks < cap ? (blocks > 0 ? blocks : 1) : cap);
    const size_t smem = gumbel_smem_bytes(L);
    const int taps = L.p.k_h * L.p.k_w;
    if (gumbel_streamed(L)) {
        const int sgrid = L.num_sms;
        if (L.p.dtype == SKIPCONV_BF16)
            gate_pixel_gumbel_stream_kernel<__nv_bfloat16><<<sgrid, GS_WARPS * 32, gumbel_stream_smem_bytes(), L.stream>>>(
                (const __nv_bfloat16*)x_t, (const __nv_bfloat16*)x_prev, (__nv_bfloat16*)x_next, chg_prev, chg_cur,
                L.gphi, L.pix_taps, n_pix, taps, step_count(L), next_count(L), L.err_dev);
        else
            gate_pixel_gumbel_stream_kernel<float><<<sgrid, GS_WARPS * 32, gumbel_stream_smem_bytes(), L.stream>>>(
                (const float*)x_t, (const float*)x_prev, (float*)x_next, chg_prev, chg_cur, L.gphi, L.pix_taps, n_pix,
                taps, step_count(L), next_count(L), L.err_dev);
        return cudaGetLastError();
    }
    const int lg = gumbel_vec_log2g(L);
    if (lg) {
        const long long per_block = 16LL * (32 >> lg);   // pixels per CTA pass (two per lane group)
        const long long vblocks = (n_pix + per_block - 1) / per_block;
        const int vgrid = (int)(vblocks < cap ? (vblocks > 0 ? vblocks : 1) : cap);
#define SC_GUMBEL_VEC(T, LG)                                                                                       \
    gate_pixel_gumbel_vec_kernel<T, LG><<<vgrid, 256, smem, L.stream>>>(                                            \
        (const T*)x_t, (const T*)x_prev, (T*)x_next, chg_prev, chg_cur, L.gphi, L.pix_taps, n_pix, L.p.c_in, taps,   \
        step_count(L), next_count(L))
        if (L.p.dtype == SKIPCONV_BF16) {
            if (lg == 5) SC_GUMBEL_VEC(__nv_bfloat16, 5);
            else if (lg == 4) SC_GUMBEL_VEC(__nv_bfloat16, 4);
            else SC_GUMBEL_VEC(__nv_bfloat16, 3);
        } else {
            if (lg == 5) SC_GUMBEL_VEC(float, 5);
            else if (lg == 4) SC_GUMBEL_VEC(float, 4);
            else SC_GUMBEL_VEC(float, 3);
        }
#undef SC_GUMBEL_VEC
        return cudaGetLastError();
    }
    if (L.p.dtype == SKIPCONV_BF16)
        gate_pixel_gumbel_kernel<__nv_bfloat16><<<grid, 256, smem, L.stream>>>(
            (const __nv_bfloat16*)x_t, (const __nv_bfloat16*)x_prev, (__nv_bfloat16*)x_next, chg_prev, chg_cur,
            L.gphi, L.pix_taps, n_pix, L.p.c_in, taps, step_count(L), next_count(L));
    else
        gate_pixel_gumbel_kernel<float><<<grid, 256, smem, L.stream>>>(
            (const float*)x_t, (const float*)x_prev, (float*)x_next, chg_prev, chg_cur, L.gphi, L.pix_taps, n_pix,
            L.p.c_in, taps, step_count(L), next_count(L));
    return cudaGetLastError();
}

cudaError_t launch_gate_blocks_gumbel(const Layer& L, int force)
{
    const GateGeom g = geom_of(L);
    const long long nblocks = (long long)L.p.n_streams * L.nby * L.nbx;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((nblocks + 7) / 8));
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = L.stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, gate_block_gumbel_kernel, (const float*)L.pix_taps, L.mask, L.list,
                              step_count(L), g, L.gate_thr, L.gphi_bias, force);
}

cudaError_t launch_gate_pixels(const Layer& L, const void* x_t, const void* x_prev, void* x_next,
                               const uint8_t* chg_prev, uint8_t* chg_cur, int force)
{
    if (L.p.dtype == SKIPCONV_BF16)
        return launch_typed<__nv_bfloat16>(L, x_t, x_prev, x_next, chg_prev, chg_cur, force);
    return launch_typed<float>(L, x_t, x_prev, x_next, chg_prev, chg_cur, force);
}

}  // namespace sc
