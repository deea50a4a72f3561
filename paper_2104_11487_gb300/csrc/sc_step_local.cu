// One-launch Skip-Conv step for small (latency-bound) layers and for layers on
// the CUDA-core path.
//
// Every CTA takes a tile of sb x sb gate blocks and does the whole step for
// it from its own input footprint (the union of the receptive fields of the
// tile's output locations):
//   1. r_t = x_t - x_{t-1} over the footprint (Eq. 2), kept in shared memory
//      as float32, and each pixel's l1 norm over all input channels;
//   2. the commit of x_t into the ping-pong buffer that becomes x_{t-1} at the
//      next step, for the input pixels this tile owns (pixels that changed at
//      this step or the previous one), and the pixels' change flags;
//   3. the block gates: per output location the norms summed over its
//      k_h x k_w receptive field (the local support norm of Eq. 5), the block
//      maximum (max-pooling of the gate, Sec. 3.2) against the threshold;
//   4. the open blocks appended to the compact list (one atomic per tile);
//   5. w * r_t at the open locations, added into z in place (Eq. 3): for dense
//      bf16 layers under SKIPCONV_PATH_AUTO a tcgen05 implicit GEMM of the
//      open locations' receptive fields (A, built in shared memory from the
//      footprints) by the slice's weights (B), accumulated in tensor memory;
//      otherwise from the shared-memory residual, a register-blocked
//      contraction over k_h*k_w*(c_in/groups) on float32 FMAs (dense and
//      grouped layers), or one thread per channel and location (depthwise);
//   6. y = act(z) at the open locations, or y = act(z + shortcut) over the
//      whole tile when the layer has a shortcut.
// Halo pixels shared with neighbouring tiles are recomputed instead of
// exchanged, so no CTA waits on another, and the launch is a programmatic
// dependent of the previous kernel in the stream (typically the layer that
// produced x_t): its CTAs are scheduled while that kernel drains and start
// reading x_t once it has completed.
//
// Two forms.  The staged form (dense layers with groups = 1, and depthwise
// layers, when a pixel's channels are a multiple of 16 bytes and at most 256)
// gives each CTA one slice of 16 or 32 output channels of a tile (depthwise: all
// channels) and moves its data with asynchronous copies: the slice's weights
// with one bulk copy issued before the dependency wait (they are constant
// state), the x_t and x_{t-1} footprints as two TMA boxes right after it
// (zero fill outside the frame is the convolution's zero padding), so that a
// step costs about three memory round trips (footprint, weights in parallel,
// z).  The contraction is split over k when the open locations are too few
// to occupy the CTA.  The general form loads with plain per-thread accesses
// and reads weights from global memory; it serves every other shape.
#include <algorithm>

#include "sc_internal.h"
#include "sc_ptx.cuh"
#include "sc_tc_common.cuh"

namespace sc {
namespace {

using namespace ptx;

constexpr int LT = 128;               // threads per CTA
constexpr int LPI = 2;                // output locations per work item of the dense contraction
constexpr int GIPT = 2;               // work items per thread and round (general form)
constexpr int GKC = 16;               // contraction chunk staged in shared memory (general form)
constexpr int MAX_TILE_BLOCKS = 16;   // sb <= 4

struct LocalArgs {
    const void* xt;
    const void* xp;            // x_{t-1}
    void* xn;                  // receives x_t (holds x_{t-2})
    const uint8_t* chg_prev;   // pixels that changed at the previous step
    uint8_t* chg_cur;          // pixels that change at this step
    const float* wcc;          // [k_h][k_w][cpg][c_out] float32
    float* z;
    void* y;                   // or NULL
    const void* sc;            // shortcut, or NULL
    uint8_t* mask;
    int32_t* list;
    int32_t* count_cur;        // this step's open-block count (zeroed by the previous step or the reset)
    int32_t* count_next;       // zeroed here for the next step
    int force;                 // key frame or dense mode: every block open
    int n, H, W, C, Ho, Wo, Co, KH, KW, stride, pad, b, nby, nbx, cpg, opg, groups, act;
    int sb, nty, ntx, FH, FW, CP;
    float thr;                 // threshold on the raw local l1 sum
    uint8_t* ychg;             // per block: this step may change y (NULL without y)
    const uint8_t* psc_chg;    // the shortcut's producer's flags (NULL: unknown, assume changed)
    int pscb, pscnby, pscnbx;
    const float* flow;         // warped residual (Eq. 10-11): [n][h][w][2] (dy, dx), or NULL
};

// The previous input as a warped residual sees it at pixel (iy, ix): T(x_{t-1})
// samples x_{t-1} at (iy + dy, ix + dx) by bilinear interpolation of the four
// surrounding pixels, a pixel outside the frame contributing zero (Eq. 10-11).
// Corner element offsets of channel 0, and their weights (0 outside).
struct Bilinear {
    size_t off[4];
    float wt[4];
};

__device__ __forceinline__ Bilinear bilinear_of(const float* flow, int nn, int H, int W, int C, int iy, int ix)
{
    const size_t pix = ((size_t)nn * H + iy) * W + ix;
    const float sy = (float)iy + flow[2 * pix], sx = (float)ix + flow[2 * pix + 1];
    const float y0f = floorf(sy), x0f = floorf(sx);
    const float ay = sy - y0f, ax = sx - x0f;
    const int y0 = (int)y0f, x0 = (int)x0f;
    const int ys[4] = {y0, y0, y0 + 1, y0 + 1}, xs[4] = {x0, x0 + 1, x0, x0 + 1};
    const float w[4] = {(1.f - ay) * (1.f - ax), (1.f - ay) * ax, ay * (1.f - ax), ay * ax};
    Bilinear b;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const bool in = ys[q] >= 0 && ys[q] < H && xs[q] >= 0 && xs[q] < W;
        b.off[q] = in ? (((size_t)nn * H + ys[q]) * W + xs[q]) * C : 0;
        b.wt[q] = in ? w[q] : 0.f;
    }
    return b;
}

template <typename T>
__device__ __forceinline__ float warped_at(const T* xp, const Bilinear& b, int c)
{
    float v = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) v += b.wt[q] * to_f32(xp[b.off[q] + c]);
    return v;
}

__device__ __forceinline__ unsigned bits_of(float v) { return __float_as_uint(v); }
__device__ __forceinline__ unsigned bits_of(__nv_bfloat16 v) { return (unsigned)__bfloat16_as_ushort(v); }

__device__ __forceinline__ float warp_sum(float v)
{
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    return v;
}

__device__ __forceinline__ float warp_max(float v)
{
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
    return v;
}

// Whether any of a producer's gate blocks over rows [r0, r1) x columns [c0, c1)
// of stream nn flagged a change (every thread of the CTA calls it; returns the
// calling thread's share, to be combined with __syncthreads_or).
__device__ __forceinline__ int any_block_flag(const uint8_t* flags, int b, int nby, int nbx, int nn, int r0, int r1,
                                              int c0, int c1, int tid, int nthreads)
{
    if (r1 <= r0 || c1 <= c0) return 0;
    const int by0 = r0 / b, bx0 = c0 / b;
    const int nbw = (c1 - 1) / b - bx0 + 1, nbb = ((r1 - 1) / b - by0 + 1) * nbw;
    int any = 0;
    for (int q = tid; q < nbb; q += nthreads)
        any |= flags[((size_t)nn * nby + by0 + q / nbw) * nbx + bx0 + q % nbw];
    return any;
}

template <typename T, bool DW, bool V4>
__global__ void __launch_bounds__(LT) step_local_kernel(const LocalArgs a)
{
    extern __shared__ __align__(16) float sm[];
    __shared__ int s_open[MAX_TILE_BLOCKS];
    __shared__ int s_nloc;
    const int FP = a.FH * a.FW;
    float* R = sm;                                   // [FP][CP] residual of the footprint
    float* P = R + (size_t)FP * a.CP;                // [FP] per-pixel l1 norm
    int* locs = reinterpret_cast<int*>(P + FP);      // open output locations of the tile, (li << 16) | lj

    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    const T* xt = static_cast<const T*>(a.xt);
    const T* xp = static_cast<const T*>(a.xp);
    T* xn = static_cast<T*>(a.xn);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int NW = LT / 32;
    const int tile = blockIdx.x;
    const int tx = tile % a.ntx, ty = (tile / a.ntx) % a.nty, nn = tile / (a.ntx * a.nty);
    const int span = a.sb * a.b;                     // output locations per tile side
    const int oy0 = ty * span, ox0 = tx * span;
    const int fy0 = oy0 * a.stride - a.pad, fx0 = ox0 * a.stride - a.pad;
    if (tile == 0 && threadIdx.x == 0) *a.count_next = 0;
    if (threadIdx.x == 0) s_nloc = 0;

    const int own_y0 = min(ty * span * a.stride, a.H);
    const int own_y1 = ty == a.nty - 1 ? a.H : min((ty + 1) * span * a.stride, a.H);
    const int own_x0 = min(tx * span * a.stride, a.W);
    const int own_x1 = tx == a.ntx - 1 ? a.W : min((tx + 1) * span * a.stride, a.W);
    const int ow = own_x1 - own_x0, npx = (own_y1 - own_y0) * ow;
    if (a.C <= 16) {
        // few channels: a thread per pixel, so that every pixel's loads are in flight at once
        // 1. residual of the footprint and per-pixel norms
        for (int q = threadIdx.x; q < FP; q += LT) {
            const int iy = fy0 + q / a.FW, ix = fx0 + q % a.FW;
            const bool in = iy >= 0 && iy < a.H && ix >= 0 && ix < a.W;
            const size_t base = in ? (((size_t)nn * a.H + iy) * a.W + ix) * a.C : 0;
            float s = 0.f;
            if (a.flow && in) {
                const Bilinear bl = bilinear_of(a.flow, nn, a.H, a.W, a.C, iy, ix);
                for (int c = 0; c < a.C; ++c) {
                    const float r = to_f32(xt[base + c]) - warped_at(xp, bl, c);
                    R[(size_t)q * a.CP + c] = r;
                    s += fabsf(r);
                }
            } else {
                for (int c = 0; c < a.C; ++c) {
                    const float r = in ? to_f32(xt[base + c]) - to_f32(xp[base + c]) : 0.f;
                    R[(size_t)q * a.CP + c] = r;
                    s += fabsf(r);
                }
            }
            P[q] = s;
        }
        // 2. commit x_t for the input pixels this tile owns (each input pixel has exactly one owner)
        for (int q = threadIdx.x; q < npx; q += LT) {
            const size_t pix = ((size_t)nn * a.H + own_y0 + q / ow) * a.W + own_x0 + q % ow;
            const size_t base = pix * a.C;
            unsigned d = 0;
            for (int c = 0; c < a.C; ++c) d |= bits_of(xt[base + c]) ^ bits_of(xp[base + c]);
            if (d || a.chg_prev[pix])
                for (int c = 0; c < a.C; ++c) xn[base + c] = xt[base + c];
            a.chg_cur[pix] = d ? 1 : 0;
        }
    } else {
        // 1. residual of the footprint and per-pixel norms (a warp per pixel, lanes over channels)
        for (int q = warp; q < FP; q += NW) {
            const int fy = q / a.FW, fx = q - (q / a.FW) * a.FW;
            const int iy = fy0 + fy, ix = fx0 + fx;
            const bool in = iy >= 0 && iy < a.H && ix >= 0 && ix < a.W;
            const size_t base = in ? (((size_t)nn * a.H + iy) * a.W + ix) * a.C : 0;
            float s = 0.f;
            if (a.flow && in) {
                const Bilinear bl = bilinear_of(a.flow, nn, a.H, a.W, a.C, iy, ix);
                for (int c = lane; c < a.C; c += 32) {
                    const float r = to_f32(xt[base + c]) - warped_at(xp, bl, c);
                    R[(size_t)q * a.CP + c] = r;
                    s += fabsf(r);
                }
            } else {
                for (int c = lane; c < a.C; c += 32) {
                    const float r = in ? to_f32(xt[base + c]) - to_f32(xp[base + c]) : 0.f;
                    R[(size_t)q * a.CP + c] = r;
                    s += fabsf(r);
                }
            }
            s = warp_sum(s);
            if (lane == 0) P[q] = s;
        }
        // 2. commit x_t for the input pixels this tile owns (each input pixel has exactly one owner)
        for (int q = warp; q < npx; q += NW) {
            const int iy = own_y0 + q / ow, ix = own_x0 + q % ow;
            const size_t pix = ((size_t)nn * a.H + iy) * a.W + ix;
            const size_t base = pix * a.C;
            unsigned d = 0;
            for (int c = lane; c < a.C; c += 32) d |= bits_of(xt[base + c]) ^ bits_of(xp[base + c]);
            const bool changed = __any_sync(0xffffffffu, d != 0);
            if (changed || a.chg_prev[pix])
                for (int c = lane; c < a.C; c += 32) xn[base + c] = xt[base + c];
            if (lane == 0) a.chg_cur[pix] = changed ? 1 : 0;
        }
    }
    __syncthreads();

    // 3. block gates of the tile (a warp per gate block)
    for (int bq = warp; bq < a.sb * a.sb; bq += NW) {
        const int bi = bq / a.sb, bj = bq - (bq / a.sb) * a.sb;
        const int by = ty * a.sb + bi, bx = tx * a.sb + bj;
        int open = 0;
        if (by < a.nby && bx < a.nbx) {
            const int bh = min(a.b, a.Ho - by * a.b), bw = min(a.b, a.Wo - bx * a.b);
            float best = -1.f;
            for (int q = lane; q < bh * bw; q += 32) {
                const int li = bi * a.b + q / bw, lj = bj * a.b + q % bw;
                float S = 0.f;
                for (int kh = 0; kh < a.KH; ++kh)
                    for (int kw = 0; kw < a.KW; ++kw) S += P[(li * a.stride + kh) * a.FW + lj * a.stride + kw];
                best = fmaxf(best, S);
            }
            best = warp_max(best);
            open = (a.force || best > a.thr) ? 1 : 0;
            if (lane == 0) {
                a.mask[((size_t)nn * a.nby + by) * a.nbx + bx] = (uint8_t)open;
                if (a.ychg) {
                    int yc = open;
                    if (!yc && a.sc)
                        yc = a.psc_chg == nullptr ? 1
                                                  : any_block_flag(a.psc_chg, a.pscb, a.pscnby, a.pscnbx, nn, by * a.b,
                                                                   min(a.Ho, (by + 1) * a.b), bx * a.b,
                                                                   min(a.Wo, (bx + 1) * a.b), 0, 1);
                    a.ychg[((size_t)nn * a.nby + by) * a.nbx + bx] = (uint8_t)(yc != 0);
                }
            }
        }
        if (lane == 0) s_open[bq] = open;
    }
    __syncthreads();

    // 4. the open blocks into the list (one atomic per tile), the open locations into shared memory
    if (warp == 0) {
        const int nb = a.sb * a.sb;
        const int o = lane < nb ? s_open[lane] : 0;
        const unsigned bal = __ballot_sync(0xffffffffu, o);
        int base = 0;
        if (lane == 0 && bal) base = atomicAdd(a.count_cur, __popc(bal));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (o) {
            const int by = ty * a.sb + lane / a.sb, bx = tx * a.sb + lane % a.sb;
            a.list[base + __popc(bal & ((1u << lane) - 1u))] = (int32_t)(((size_t)nn * a.nby + by) * a.nbx + bx);
        }
    }
    for (int q = threadIdx.x; q < span * span; q += LT) {
        const int li = q / span, lj = q - (q / span) * span;
        if (s_open[(li / a.b) * a.sb + lj / a.b] && oy0 + li < a.Ho && ox0 + lj < a.Wo)
            locs[atomicAdd(&s_nloc, 1)] = (li << 16) | lj;
    }
    __syncthreads();

    // 5. w * r_t at the open locations into z (and y = act(z) when there is no shortcut)
    const int M = s_nloc;
    T* y = static_cast<T*>(a.y);
    const bool y_here = y != nullptr && a.sc == nullptr;
    if (DW) {
        for (int it = threadIdx.x; it < M * a.C; it += LT) {
            const int c = it % a.C, m = it / a.C;
            const int loc = locs[m], li = loc >> 16, lj = loc & 0xffff;
            const float* r = R + (size_t)(li * a.stride * a.FW + lj * a.stride) * a.CP + c;
            float acc = 0.f;
            for (int kh = 0; kh < a.KH; ++kh)
                for (int kw = 0; kw < a.KW; ++kw)
                    acc = fmaf(__ldg(a.wcc + (size_t)(kh * a.KW + kw) * a.Co + c), r[(size_t)(kh * a.FW + kw) * a.CP],
                               acc);
            const size_t zo = (((size_t)nn * a.Ho + oy0 + li) * a.Wo + ox0 + lj) * a.Co + c;
            const float zv = a.z[zo] + acc;
            a.z[zo] = zv;
            if (y_here) y[zo] = from_f32<T>(activate(zv, a.act));
        }
    } else {
        // rounds of up to IPT work items per thread; k in chunks of GKC whose weights (all output
        // channels) and footprint offsets are staged in shared memory by the whole CTA
        const int nq = (a.opg + 3) >> 2;             // output-channel quads per group
        const int nm = (M + LPI - 1) / LPI;
        const int items = nm * a.groups * nq;
        const int K = a.KH * a.KW * a.cpg;           // contraction length of one output channel
        // [GKC][Co], 16-byte aligned for the quad loads
        float* Wc = sm + (((size_t)FP * a.CP + FP + (size_t)span * span + 3) & ~(size_t)3);
        int* toffs = reinterpret_cast<int*>(Wc + GKC * a.Co);      // [GKC] residual offset of k in the footprint
        for (int it0 = 0; it0 < items; it0 += LT * GIPT) {
            int o[GIPT], oend[GIPT], rb[GIPT][LPI];
            long long zl[GIPT][LPI];
            float acc[GIPT][LPI][4];
#pragma unroll
            for (int j = 0; j < GIPT; ++j) {
                const int it = it0 + (int)threadIdx.x + j * LT;
                const bool on = it < items;
                const int q = on ? it % nq : 0;
                const int rest = on ? it / nq : 0;
                const int grp = rest % a.groups, mi = rest / a.groups;
                o[j] = grp * a.opg + q * 4;
                oend[j] = on ? grp * a.opg + a.opg : 0;   // 0: no work
#pragma unroll
                for (int u = 0; u < LPI; ++u) {
                    const int m = mi * LPI + u;
                    if (on && m < M) {
                        const int loc = locs[m], li = loc >> 16, lj = loc & 0xffff;
                        rb[j][u] = (li * a.stride * a.FW + lj * a.stride) * a.CP + grp * a.cpg;
                        zl[j][u] = ((long long)nn * a.Ho + oy0 + li) * a.Wo + ox0 + lj;
                    } else {
                        rb[j][u] = 0;
                        zl[j][u] = -1;
                    }
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[j][u][e] = 0.f;
                }
            }
            for (int k0 = 0; k0 < K; k0 += GKC) {
                const int kc = min(GKC, K - k0);
                __syncthreads();   // the previous chunk has been used
                for (int e = threadIdx.x; e < kc * a.Co; e += LT) Wc[e] = __ldg(a.wcc + (size_t)k0 * a.Co + e);
                if ((int)threadIdx.x < kc) {
                    const int k = k0 + (int)threadIdx.x, tap = k / a.cpg, ci = k - tap * a.cpg;
                    toffs[threadIdx.x] = ((tap / a.KW) * a.FW + tap % a.KW) * a.CP + ci;
                }
                __syncthreads();
                for (int kk = 0; kk < kc; ++kk) {
                    const int toff = toffs[kk];
                    const float* wrow = Wc + kk * a.Co;
#pragma unroll
                    for (int j = 0; j < GIPT; ++j) {
                        if (oend[j] == 0) continue;
                        float4 w;
                        if (V4) {
                            w = *reinterpret_cast<const float4*>(wrow + o[j]);
                        } else {
                            w.x = wrow[o[j]];
                            w.y = o[j] + 1 < oend[j] ? wrow[o[j] + 1] : 0.f;
                            w.z = o[j] + 2 < oend[j] ? wrow[o[j] + 2] : 0.f;
                            w.w = o[j] + 3 < oend[j] ? wrow[o[j] + 3] : 0.f;
                        }
#pragma unroll
                        for (int u = 0; u < LPI; ++u) {
                            const float r = R[rb[j][u] + toff];
                            acc[j][u][0] = fmaf(r, w.x, acc[j][u][0]);
                            acc[j][u][1] = fmaf(r, w.y, acc[j][u][1]);
                            acc[j][u][2] = fmaf(r, w.z, acc[j][u][2]);
                            acc[j][u][3] = fmaf(r, w.w, acc[j][u][3]);
                        }
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < GIPT; ++j) {
#pragma unroll
                for (int u = 0; u < LPI; ++u) {
                    if (zl[j][u] < 0) continue;
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        if (o[j] + e >= oend[j]) continue;
                        const size_t zo = (size_t)zl[j][u] * a.Co + o[j] + e;
                        const float zv = a.z[zo] + acc[j][u][e];
                        a.z[zo] = zv;
                        if (y_here) y[zo] = from_f32<T>(activate(zv, a.act));
                    }
                }
            }
        }
    }

    // 6. with a shortcut: y = act(z + shortcut) over the tile's output locations
    if (y != nullptr && a.sc != nullptr) {
        __syncthreads();   // this CTA's z updates are visible to all its threads
        const T* sc = static_cast<const T*>(a.sc);
        const int th = min(span, a.Ho - oy0), tw = min(span, a.Wo - ox0);
        for (int it = threadIdx.x; it < th * tw * a.Co; it += LT) {
            const int c = it % a.Co, p = it / a.Co;
            const size_t zo = (((size_t)nn * a.Ho + oy0 + p / tw) * a.Wo + ox0 + p % tw) * a.Co + c;
            y[zo] = from_f32<T>(activate(a.z[zo] + to_f32(sc[zo]), a.act));
        }
    }
}

// ------------------------------------------------------------- staged form
constexpr int FT = 256;                          // threads per CTA
constexpr int SW_WIDE = 32, SW_NARROW = 16;       // output channels per CTA (dense layers)
constexpr int FLPI = 2;                          // output locations per work item
constexpr uint64_t LOCAL_WAIT_NS = 1000000000ull;

struct FastArgs {
    const void* wpack;         // dense: [slice][K][SW]; depthwise: [taps][C] (layer dtype)
    uint32_t wbytes;           // weight bytes of one CTA (a multiple of 16)
    const void* xt;            // x_t and x_{t-1} in global memory (owned pixels outside the footprint)
    const void* xp;
    void* xn;
    const uint8_t* chg_prev;
    uint8_t* chg_cur;
    float* z;
    void* y;
    const void* sc;
    uint8_t* mask;
    int32_t* list;
    int32_t* count_cur;
    int32_t* count_next;
    int* err;
    int force;
    int n, H, W, C, Ho, Wo, Co, KH, KW, stride, pad, b, nby, nbx, act;
    int sb, nty, ntx, FH, FW, CP, nsl, K;
    int Kp;                    // tensor-core contraction: K rounded up to 16 (the MMA's K step)
    uint32_t off_xp, off_w, off_r, off_p, off_loc, off_scr, off_z, off_sc, off_chg, off_dq;   // byte offsets
    uint32_t off_a;            // tensor-core contraction: the A region (its last 2 KB stay free)
    int aregion;               //   and its size in bytes
    float thr;
    // stack propagation
    const uint8_t* px_chg;       // the layer that produced x_t: its per-block "y may have changed" flags
    int pxb, pxnby, pxnbx;       //   (NULL when x_t is not a linked layer's y of the step just before)
    const uint8_t* psc_chg;      // the same for the shortcut's producer
    int pscb, pscnby, pscnbx;
    uint8_t* ychg;               // this layer's per-block y-change flags (NULL without y)
    const uint8_t* tile_chg_prev;  // per tile: some owned pixel changed at the previous step
    uint8_t* tile_chg_cur;       // per tile: some owned pixel changes at this step
};



__device__ __forceinline__ float4 load_w4(const float* w) { return *reinterpret_cast<const float4*>(w); }
__device__ __forceinline__ float4 load_w4(const __nv_bfloat16* w)
{
    const uint2 v = *reinterpret_cast<const uint2*>(w);
    const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&v.x));
    const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&v.y));
    return make_float4(lo.x, lo.y, hi.x, hi.y);
}

// Residuals of one 16-byte chunk of a pixel (8 bf16 or 4 fp32 channels),
// their l1 sum, and whether any bit differs.
__device__ __forceinline__ int chunk_residual(const uint4& a, const uint4& b, float (&r)[8], __nv_bfloat16*)
{
    const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
    const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 fa = __bfloat1622float2(pa[k]), fb = __bfloat1622float2(pb[k]);
        r[2 * k] = fa.x - fb.x;
        r[2 * k + 1] = fa.y - fb.y;
    }
    return 8;
}

__device__ __forceinline__ int chunk_residual(const uint4& a, const uint4& b, float (&r)[8], float*)
{
    r[0] = __uint_as_float(a.x) - __uint_as_float(b.x);
    r[1] = __uint_as_float(a.y) - __uint_as_float(b.y);
    r[2] = __uint_as_float(a.z) - __uint_as_float(b.z);
    r[3] = __uint_as_float(a.w) - __uint_as_float(b.w);
    return 4;
}

// x_t's chunk minus the matching fp32 values of the warped previous input.
__device__ __forceinline__ int chunk_minus_f32(const uint4& a, const float* w, float (&r)[8], __nv_bfloat16*)
{
    const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
    const float4 w0 = reinterpret_cast<const float4*>(w)[0], w1 = reinterpret_cast<const float4*>(w)[1];
    const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 fa = __bfloat1622float2(pa[k]);
        r[2 * k] = fa.x - wv[2 * k];
        r[2 * k + 1] = fa.y - wv[2 * k + 1];
    }
    return 8;
}

__device__ __forceinline__ int chunk_minus_f32(const uint4& a, const float* w, float (&r)[8], float*)
{
    const float4 w0 = reinterpret_cast<const float4*>(w)[0];
    r[0] = __uint_as_float(a.x) - w0.x;
    r[1] = __uint_as_float(a.y) - w0.y;
    r[2] = __uint_as_float(a.z) - w0.z;
    r[3] = __uint_as_float(a.w) - w0.w;
    return 4;
}

__device__ __forceinline__ float2 load_pair(const float* p) { return *reinterpret_cast<const float2*>(p); }
__device__ __forceinline__ float2 load_pair(const __nv_bfloat16* p)
{
    return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p));
}

// Eight fp32 values as eight bf16 (round to nearest even), in memory order.
__device__ __forceinline__ uint4 pack_bf16x8(const float4& a, const float4& b)
{
    uint4 v;
    __nv_bfloat162 h[4] = {__floats2bfloat162_rn(a.x, a.y), __floats2bfloat162_rn(a.z, a.w),
                           __floats2bfloat162_rn(b.x, b.y), __floats2bfloat162_rn(b.z, b.w)};
    v.x = *reinterpret_cast<uint32_t*>(&h[0]);
    v.y = *reinterpret_cast<uint32_t*>(&h[1]);
    v.z = *reinterpret_cast<uint32_t*>(&h[2]);
    v.w = *reinterpret_cast<uint32_t*>(&h[3]);
    return v;
}

constexpr int TC_ROWS = 128;                // MMA rows (open locations) per pass
// TMEM columns of the accumulator: the slice's output channels (a power of 2, at least 32)
template <int SW>
constexpr uint32_t tc_cols() { return SW < 32 ? 32u : (uint32_t)SW; }
constexpr int TC_MAX_KG = 9 * 256 / 8;      // k-groups of w in the offset table (3x3, 256 channels)
// The plain step's A: [x_t | -x_{t-1}] (exact in bf16, each half against w) when true; else
// r = x_t - x_{t-1} rounded to bf16 (one half).
constexpr bool TC_EXACT = true;
constexpr int TC_AREGION_MAX = 32 * 1024;   // most shared memory for A (its last 2 KB stay free)

template <typename T, bool DW, int SW, bool WP, bool TC>
__global__ void __launch_bounds__(FT, 1) step_local_staged_kernel(const __grid_constant__ CUtensorMap tm_xt,
                                                               const __grid_constant__ CUtensorMap tm_xp,
                                                               const __grid_constant__ CUtensorMap tm_z,
                                                               const __grid_constant__ CUtensorMap tm_sc,
                                                               const FastArgs a)
{
    static_assert(!TC || (!DW && sizeof(T) == 2), "the tensor-core contraction takes dense bf16 layers");
    extern __shared__ uint8_t smem_raw[];
    // 0: weights, 1: footprints, 2: z (and shortcut) tile, 3-4: MMAs done reading A buffer 0 / 1
    __shared__ __align__(8) uint64_t bars[5];
    __shared__ uint32_t s_tmem;
    __shared__ int s_open[MAX_TILE_BLOCKS];
    __shared__ int s_max[MAX_TILE_BLOCKS];      // per gate block: largest support sum (float bits)
    __shared__ int s_nloc;
    __shared__ int s_tchg;                      // some owned pixel changed at this step
    uint8_t* base = align_smem_1024(smem_raw);
    const T* Xt = reinterpret_cast<const T*>(base);
    const T* Xp = reinterpret_cast<const T*>(base + a.off_xp);
    const float* Xw = reinterpret_cast<const float*>(base + a.off_xp);   // WP: the warped previous input, fp32
    const T* Ws = reinterpret_cast<const T*>(base + a.off_w);
    float* R = reinterpret_cast<float*>(base + a.off_r);      // dense only: [FP][CP] residual
    float* P = reinterpret_cast<float*>(base + a.off_p);
    int* locs = reinterpret_cast<int*>(base + a.off_loc);
    float* red = reinterpret_cast<float*>(base + a.off_scr);  // dense: k-split partial sums (scratch)
    uint8_t* Dq = base + a.off_dq;                            // per footprint pixel: changed
    const float* Zs = reinterpret_cast<const float*>(base + a.off_z);   // [span*span][ZW] z of the tile
    const T* Ss = reinterpret_cast<const T*>(base + a.off_sc);          // [span*span][ZW] shortcut of the tile
    uint8_t* chgs = base + a.off_chg;                                   // owned pixels' previous change flags
    constexpr int ZW = DW ? 0 : SW;                                     // channels of the z tile (dense)
    const int zw = DW ? a.Co : ZW;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    constexpr int NW = FT / 32;
    const int sl = DW ? 0 : (int)(blockIdx.x % a.nsl);
    const int tile = DW ? (int)blockIdx.x : (int)(blockIdx.x / a.nsl);
    const int tx = tile % a.ntx, ty = (tile / a.ntx) % a.nty, nn = tile / (a.ntx * a.nty);
    const int span = a.sb * a.b;
    const int oy0 = ty * span, ox0 = tx * span;
    const int fy0 = oy0 * a.stride - a.pad, fx0 = ox0 * a.stride - a.pad;
    const int FP = a.FH * a.FW;
    const int o_base = DW ? 0 : sl * SW;
    const bool has_sc = a.sc != nullptr;
    const uint32_t bar_w = smem_u32(&bars[0]), bar_x = smem_u32(&bars[1]), bar_z = smem_u32(&bars[2]);
    const uint32_t ztx = (uint32_t)(span * span * zw) * (4u + (has_sc ? (uint32_t)sizeof(T) : 0u));

    if (tid == 0) {
        mbar_init(bar_w, 1);
        mbar_init(bar_x, 1);
        mbar_init(bar_z, 1);
        if (TC) {
            mbar_init(smem_u32(&bars[3]), 1);
            mbar_init(smem_u32(&bars[4]), 1);
        }
        fence_mbar_init();
        // the weights are constant state: fetch them before waiting for the producer of x_t
        mbar_arrive_expect_tx(bar_w, a.wbytes);
        bulk_load(smem_u32(Ws), static_cast<const uint8_t*>(a.wpack) + (size_t)sl * a.wbytes, a.wbytes, bar_w);
        prefetch_tmap(&tm_xt);
        prefetch_tmap(&tm_xp);
        s_nloc = 0;
        s_tchg = 0;
    }
    if (tid < MAX_TILE_BLOCKS) s_max[tid] = 0;
    if (TC) {
        // the accumulator's 32 TMEM columns, taken while the previous grid finishes.  The grid that
        // launched this one early had every CTA take its columns before it let this grid start, and
        // a grid after this one starts only once every CTA here passed the dependency wait, so at
        // most two grids hold columns on an SM: at most 8 CTAs of 256 threads, 256 of 512 columns,
        // and an allocation here never waits for a CTA that waits for this grid.
        if (warp == 0) {
            tmem_alloc(smem_u32(&s_tmem), tc_cols<SW>());
            tmem_relinquish();
        }
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
    }
    grid_dependency_wait();
    if (blockIdx.x == 0 && tid == 0) *a.count_next = 0;
    // owned input pixels of this tile (every input pixel has exactly one owner tile)
    const int own_y0 = min(ty * span * a.stride, a.H);
    const int own_y1 = ty == a.nty - 1 ? a.H : min((ty + 1) * span * a.stride, a.H);
    const int own_x0 = min(tx * span * a.stride, a.W);
    const int own_x1 = tx == a.ntx - 1 ? a.W : min((tx + 1) * span * a.stride, a.W);
    const int oww = own_x1 - own_x0, npx = (own_y1 - own_y0) * oww;
    if (a.px_chg != nullptr && !a.force) {
        // stack propagation: x_t is a linked layer's y, which changed only in the blocks that layer
        // flagged.  If none under this tile's footprint and owned pixels changed, no owned pixel
        // changed at the previous step either, and the shortcut did not change over the tile, then
        // r_t = 0 over the footprint: every block stays closed and there is nothing to commit or
        // refresh -- the full step's outcome, without reading the tile.
        int any = (tid == 0 && a.tile_chg_prev[tile]) ? 1 : 0;
        any |= any_block_flag(a.px_chg, a.pxb, a.pxnby, a.pxnbx, nn, max(0, min(fy0, own_y0)),
                              min(a.H, max(fy0 + a.FH, own_y1)), max(0, min(fx0, own_x0)),
                              min(a.W, max(fx0 + a.FW, own_x1)), tid, FT);
        if (has_sc) {
            if (a.psc_chg == nullptr) any = 1;
            else any |= any_block_flag(a.psc_chg, a.pscb, a.pscnby, a.pscnbx, nn, oy0, min(a.Ho, oy0 + span), ox0,
                                       min(a.Wo, ox0 + span), tid, FT);
        }
        if (!__syncthreads_or(any)) {
            if (sl == 0) {
                for (int bq = tid; bq < a.sb * a.sb; bq += FT) {
                    const int by = ty * a.sb + bq / a.sb, bx = tx * a.sb + bq % a.sb;
                    if (by < a.nby && bx < a.nbx) {
                        a.mask[((size_t)nn * a.nby + by) * a.nbx + bx] = 0;
                        if (a.ychg) a.ychg[((size_t)nn * a.nby + by) * a.nbx + bx] = 0;
                    }
                }
                if (a.tile_chg_cur[tile]) {   // this parity's flags still hold two steps ago's changes
                    for (int q = tid; q < npx; q += FT)
                        a.chg_cur[((size_t)nn * a.H + own_y0 + q / oww) * a.W + own_x0 + q % oww] = 0;
                    if (tid == 0) a.tile_chg_cur[tile] = 0;
                }
            }
            if (tid == 0) mbar_wait(bar_w, 0, nullptr, nullptr, LOCAL_WAIT_NS);   // the weight copy in flight
            if (TC && warp == 0) tmem_dealloc(s_tmem, tc_cols<SW>());
            return;
        }
    }
    if (tid == 0) {
        mbar_arrive_expect_tx(bar_x, (uint32_t)FP * (uint32_t)a.C * (uint32_t)(sizeof(T) + (WP ? 4 : sizeof(T))));
        tma_load_4d(smem_u32(Xt), &tm_xt, bar_x, 0, fx0, fy0, nn);
        tma_load_4d(smem_u32(Xp), &tm_xp, bar_x, 0, fx0, fy0, nn);
        if (has_sc) {
            // with a shortcut every location's y is refreshed: z and the shortcut of the whole tile
            mbar_arrive_expect_tx(bar_z, ztx);
            tma_load_4d(smem_u32(Zs), &tm_z, bar_z, o_base, ox0, oy0, nn);
            tma_load_4d(smem_u32(Ss), &tm_sc, bar_z, o_base, ox0, oy0, nn);
        }
    }
    grid_launch_dependents();

    // slice 0: the owned pixels' change flags of the previous step
    if (sl == 0)
        for (int q = tid; q < npx; q += FT)
            chgs[q] = a.chg_prev[((size_t)nn * a.H + own_y0 + q / oww) * a.W + own_x0 + q % oww];
    __syncthreads();   // barrier initialisation and the flags visible to every thread
    {
        const bool ok = mbar_wait(bar_x, 0, nullptr, a.err, LOCAL_WAIT_NS);
        if (!__syncthreads_and(ok)) {
            // copies may still be in flight into this CTA's shared memory: wait for them (bounded) first
            mbar_wait(bar_x, 0, nullptr, nullptr, LOCAL_WAIT_NS);
            mbar_wait(bar_w, 0, nullptr, nullptr, LOCAL_WAIT_NS);
            if (has_sc) mbar_wait(bar_z, 0, nullptr, nullptr, LOCAL_WAIT_NS);
            if (TC && warp == 0) tmem_dealloc(s_tmem, tc_cols<SW>());
            return;
        }
    }
    T* xn = static_cast<T*>(a.xn);

    // residuals, per-chunk partial norms and change bits: one thread per (footprint pixel, 16-byte chunk)
    constexpr int EPC = 16 / (int)sizeof(T);
    const int CH = a.C / EPC;
    {
        float* Pp = reinterpret_cast<float*>(base + a.off_scr);            // [FP][CH]
        uint8_t* Dp = base + a.off_scr + (size_t)FP * CH * sizeof(float);   // [FP][CH]
        for (int it = tid; it < FP * CH; it += FT) {
            const int q = it / CH, k = it - (it / CH) * CH;
            const uint4 av = reinterpret_cast<const uint4*>(Xt + (size_t)q * a.C)[k];
            float r[8];
            int ne;
            if (WP) {
                // r_t = x_t - T(x_{t-1}) (Eq. 10-11); the commit compared the raw frames in the pre-pass
                ne = chunk_minus_f32(av, Xw + (size_t)q * a.C + k * EPC, r, (T*)nullptr);
                Dp[it] = 0;
            } else {
                const uint4 bv = reinterpret_cast<const uint4*>(Xp + (size_t)q * a.C)[k];
                ne = chunk_residual(av, bv, r, (T*)nullptr);
                Dp[it] = ((av.x ^ bv.x) | (av.y ^ bv.y) | (av.z ^ bv.z) | (av.w ^ bv.w)) != 0u;
            }
            float sum = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e)
                if (e < ne) sum += fabsf(r[e]);
            Pp[it] = sum;
            if (!DW && (!TC || WP)) {   // the fp32 residual feeds the FMA contraction and the warped step's A
                float4* rr = reinterpret_cast<float4*>(R + (size_t)q * a.CP + k * EPC);
                rr[0] = make_float4(r[0], r[1], r[2], r[3]);
                if (EPC == 8) rr[1] = make_float4(r[4], r[5], r[6], r[7]);
            }
        }
        __syncthreads();
        // per pixel: the l1 norm (chunk partials in channel order) and whether any bit changed
        for (int q = tid; q < FP; q += FT) {
            float sum = 0.f;
            unsigned d = 0;
            for (int k = 0; k < CH; ++k) {
                sum += Pp[q * CH + k];
                d |= Dp[q * CH + k];
            }
            P[q] = sum;
            Dq[q] = (uint8_t)d;
        }
    }
    __syncthreads();

    // slice 0: the commit of x_t for the owned pixels (one thread per pixel and chunk inside the
    // footprint, a warp per pixel outside it), and the pixels' change flags (WP: done by the pre-pass)
    if (sl == 0 && !WP) {
        for (int it = tid; it < npx * CH; it += FT) {
            const int q = it / CH, k = it - (it / CH) * CH;
            const int iy = own_y0 + q / oww, ix = own_x0 + q % oww;
            const int fy = iy - fy0, fx = ix - fx0;
            if (fy >= a.FH || fx >= a.FW) continue;
            const int fq = fy * a.FW + fx;
            const size_t pix = ((size_t)nn * a.H + iy) * a.W + ix;
            const bool changed = Dq[fq] != 0;
            if (changed || chgs[q])
                (reinterpret_cast<uint4*>(xn) + pix * CH)[k] = reinterpret_cast<const uint4*>(Xt + (size_t)fq * a.C)[k];
            if (k == 0) {
                a.chg_cur[pix] = changed ? 1 : 0;
                if (changed) s_tchg = 1;
            }
        }
        const T* xt = static_cast<const T*>(a.xt);
        const T* xp = static_cast<const T*>(a.xp);
        for (int q = warp; q < npx; q += NW) {
            const int iy = own_y0 + q / oww, ix = own_x0 + q % oww;
            if (iy - fy0 < a.FH && ix - fx0 < a.FW) continue;   // done from the footprint
            const size_t pix = ((size_t)nn * a.H + iy) * a.W + ix;
            unsigned d = 0;
            for (int c = lane; c < a.C; c += 32) d |= bits_of(xt[pix * a.C + c]) ^ bits_of(xp[pix * a.C + c]);
            const bool changed = __any_sync(0xffffffffu, d != 0);
            if (changed || chgs[q])
                for (int c = lane; c < a.C; c += 32) xn[pix * a.C + c] = xt[pix * a.C + c];
            if (lane == 0) {
                a.chg_cur[pix] = changed ? 1 : 0;
                if (changed) s_tchg = 1;
            }
        }
    }

    // block gates: per output location its support sum, per block the maximum (the sums are
    // non-negative, so their float bits order like integers)
    for (int q = tid; q < span * span; q += FT) {
        const int li = q / span, lj = q - (q / span) * span;
        if (oy0 + li >= a.Ho || ox0 + lj >= a.Wo) continue;
        const float* Pl = P + li * a.stride * a.FW + lj * a.stride;
        float S = 0.f;
        if (a.KH == 3 && a.KW == 3) {   // the same order, with the nine loads issued together
            float v[9];
#pragma unroll
            for (int t = 0; t < 9; ++t) v[t] = Pl[(t / 3) * a.FW + t % 3];
#pragma unroll
            for (int t = 0; t < 9; ++t) S += v[t];
        } else {
            for (int kh = 0; kh < a.KH; ++kh)
                for (int kw = 0; kw < a.KW; ++kw) S += Pl[kh * a.FW + kw];
        }
        atomicMax(&s_max[(li / a.b) * a.sb + lj / a.b], __float_as_int(S));
    }
    __syncthreads();
    if (tid < a.sb * a.sb) {
        const int by = ty * a.sb + tid / a.sb, bx = tx * a.sb + tid % a.sb;
        int open = 0;
        if (by < a.nby && bx < a.nbx) {
            open = (a.force || __int_as_float(s_max[tid]) > a.thr) ? 1 : 0;
            if (sl == 0) a.mask[((size_t)nn * a.nby + by) * a.nbx + bx] = (uint8_t)open;
        }
        s_open[tid] = open;
        // this layer's y may change where a block is open, or (with a shortcut) where the shortcut did
        if (sl == 0 && a.ychg && by < a.nby && bx < a.nbx) {
            int yc = open;
            if (!yc && has_sc)
                yc = a.psc_chg == nullptr
                         ? 1
                         : any_block_flag(a.psc_chg, a.pscb, a.pscnby, a.pscnbx, nn, by * a.b, min(a.Ho, (by + 1) * a.b),
                                          bx * a.b, min(a.Wo, (bx + 1) * a.b), 0, 1);
            a.ychg[((size_t)nn * a.nby + by) * a.nbx + bx] = (uint8_t)(yc != 0);
        }
    }
    __syncthreads();
    if (sl == 0 && tid == 0) a.tile_chg_cur[tile] = (uint8_t)s_tchg;
    bool any_open = false;
    for (int bq = 0; bq < a.sb * a.sb; ++bq) any_open |= s_open[bq] != 0;
    if (tid == 0 && any_open && !has_sc) {
        // the z tile of a tile with open blocks (without a shortcut only those are touched)
        mbar_arrive_expect_tx(bar_z, ztx);
        tma_load_4d(smem_u32(Zs), &tm_z, bar_z, o_base, ox0, oy0, nn);
    }
    // the open blocks into the list: the slot comes back while the convolution runs
    int list_base = 0, list_open = 0;
    unsigned list_bal = 0;
    if (sl == 0 && warp == 0) {
        list_open = lane < a.sb * a.sb ? s_open[lane] : 0;
        list_bal = __ballot_sync(0xffffffffu, list_open);
        if (lane == 0 && list_bal) list_base = atomicAdd(a.count_cur, __popc(list_bal));
    }
    for (int q = tid; q < span * span; q += FT) {
        const int li = q / span, lj = q - (q / span) * span;
        if (s_open[(li / a.b) * a.sb + lj / a.b] && oy0 + li < a.Ho && ox0 + lj < a.Wo)
            locs[atomicAdd(&s_nloc, 1)] = (li << 16) | lj;
    }
    {
        bool ok = mbar_wait(bar_w, 0, nullptr, a.err, LOCAL_WAIT_NS);
        if (any_open || has_sc) ok = ok && mbar_wait(bar_z, 0, nullptr, a.err, LOCAL_WAIT_NS);
        if (!__syncthreads_and(ok)) {
            mbar_wait(bar_w, 0, nullptr, nullptr, LOCAL_WAIT_NS);
            if (any_open || has_sc) mbar_wait(bar_z, 0, nullptr, nullptr, LOCAL_WAIT_NS);
            if (TC && warp == 0) tmem_dealloc(s_tmem, tc_cols<SW>());
            return;
        }
    }

    const int M = s_nloc;
    T* y = static_cast<T*>(a.y);
    auto y_of = [&](float zv, int zi) {   // the layer output at tile element zi (location * zw + channel)
        return from_f32<T>(activate(has_sc ? zv + to_f32(Ss[zi]) : zv, a.act));
    };
    if (DW) {
        // a thread per channel pair (weights in registers) and a share of the open locations
        const int NCP = a.C / 2, ngrp = FT / NCP;
        const int cp = tid % NCP, g = tid / NCP, c = 2 * cp;
        float2 wreg[9];   // 3x3 layers: the channel pair's weights
#pragma unroll
        for (int tp = 0; tp < 9; ++tp)
            wreg[tp] = (a.KH == 3 && a.KW == 3) ? load_pair(Ws + tp * a.C + c) : make_float2(0.f, 0.f);
        if (g < ngrp) {
            for (int m = g; m < M; m += ngrp) {
                const int loc = locs[m], li = loc >> 16, lj = loc & 0xffff;
                const int p0 = li * a.stride * a.FW + lj * a.stride;
                float acc0 = 0.f, acc1 = 0.f;
                if (a.KH == 3 && a.KW == 3) {
#pragma unroll
                    for (int kh = 0; kh < 3; ++kh)
#pragma unroll
                        for (int kw = 0; kw < 3; ++kw) {
                            const size_t e = (size_t)(p0 + kh * a.FW + kw) * a.C + c;
                            const float2 xa = load_pair(Xt + e);
                            const float2 xb = WP ? *reinterpret_cast<const float2*>(Xw + e) : load_pair(Xp + e);
                            acc0 = fmaf(wreg[kh * 3 + kw].x, xa.x - xb.x, acc0);
                            acc1 = fmaf(wreg[kh * 3 + kw].y, xa.y - xb.y, acc1);
                        }
                } else {
                    for (int kh = 0; kh < a.KH; ++kh)
                        for (int kw = 0; kw < a.KW; ++kw) {
                            const size_t e = (size_t)(p0 + kh * a.FW + kw) * a.C + c;
                            const float2 xa = load_pair(Xt + e);
                            const float2 xb = WP ? *reinterpret_cast<const float2*>(Xw + e) : load_pair(Xp + e);
                            const float2 w = load_pair(Ws + (kh * a.KW + kw) * a.C + c);
                            acc0 = fmaf(w.x, xa.x - xb.x, acc0);
                            acc1 = fmaf(w.y, xa.y - xb.y, acc1);
                        }
                }
                const int zi = (li * span + lj) * zw + c;
                const float z0 = Zs[zi] + acc0, z1 = Zs[zi + 1] + acc1;
                const size_t zo = (((size_t)nn * a.Ho + oy0 + li) * a.Wo + ox0 + lj) * a.Co + c;
                *reinterpret_cast<float2*>(a.z + zo) = make_float2(z0, z1);
                if (y) {
                    const T y0 = y_of(z0, zi), y1 = y_of(z1, zi + 1);
                    y[zo] = y0;
                    y[zo + 1] = y1;
                }
            }
        }
    } else if (TC) {
        // The contraction on the tensor cores (tcgen05, bf16 operands, fp32 accumulation), in
        // passes of up to 128 open locations: D[m][o] = sum_k A[m][k] B[o][k].  Row m of A is the
        // m-th open location's receptive field, k = tap * C + ci over K (padded to Kp, a multiple
        // of 16).  A plain step takes w * r_t as w * x_t + w * (-x_{t-1}) (Eq. 3 is linear in r):
        // A is [x_t | -x_{t-1}], both halves exact in bf16 and each multiplied by B = w, so the
        // products are exact and only the fp32 sums round.  A warped step's previous input
        // T(x_{t-1}) is not bf16: there A is r = x_t - T(x_{t-1}) rounded to bf16 (one half).
        // B is the slice's weights, staged by the bulk copy.  Both operands use the
        // no-swizzle K-major layout of core matrices (8 rows x 16 bytes, rows 16 bytes apart, row
        // groups 128 bytes apart): B as [k/8][SW][8]; A as [k/8][R][8] with R the pass's rows
        // rounded up to 8, so that A holds only the open locations.  An MMA reads 128 rows: rows
        // past R fall on the next k-group or on the 2 KB kept free past the A region, and only
        // feed rows of D that are not read.  A is built in one go where it fits in the region,
        // else in chunks of k-groups into two buffers (the MMAs of one chunk run while the next
        // is built).  D: TMEM lane m, columns 0..SW-1 (taken after the dependency wait).
        const uint32_t tmem = s_tmem;
        bool ok = true;
        if (M > 0) {
            const uint32_t bm0 = smem_u32(&bars[3]), bm1 = smem_u32(&bars[4]);
            uint8_t* Abuf = base + a.off_a;
            const uint8_t* Wb = reinterpret_cast<const uint8_t*>(Ws);
            const int hkg = a.Kp / 8;                                  // k-groups of w (even)
            const int tkg = (!WP && TC_EXACT) ? 2 * hkg : hkg;         // k-groups of A (even)
            // per k-group of A (8 consecutive k): its element offset from a row's first footprint
            // pixel, bit 31 set for x_{t-1}; per row of a pass: that pixel's element offset.  Both in
            // the k-split scratch, which the tensor-core contraction does not use.
            const int px = WP ? a.CP : a.C;   // elements per footprint pixel of A's source
            int* koff = reinterpret_cast<int*>(base + a.off_scr);
            int* rofs = koff + TC_MAX_KG;
            for (int kg = tid; kg < hkg; kg += FT) {
                const int k = kg * 8;   // a k-group of 8 never straddles two taps: C is a multiple of 8
                const int tap = k / a.C, ci = k - tap * a.C;
                const int kh = tap / a.KW, kw = tap - kh * a.KW;
                koff[kg] = k < a.K ? (kh * a.FW + kw) * px + ci : -1;   // -1: padding past K
            }
            constexpr uint32_t idesc = idesc_bf16_f32(TC_ROWS, SW);
            uint32_t phase = 0u;   // bit b: the next phase to wait for on buffer b's barrier
            uint32_t pend = 0u;    // bit b: MMAs reading buffer b were committed and not yet waited for
            // wait for the MMAs that read buffer b (bounded; the error word records a timeout)
            auto drain = [&](int b) {
                if (pend & (1u << b)) {
                    ok = mbar_wait(b ? bm1 : bm0, (phase >> b) & 1u, nullptr, a.err, LOCAL_WAIT_NS) && ok;
                    phase ^= 1u << b;
                    pend &= ~(1u << b);
                }
            };
            for (int m0 = 0; m0 < M && ok; m0 += TC_ROWS) {
                const int mr = min(TC_ROWS, M - m0);
                const int rb = ((mr + 7) & ~7) * 16;                       // bytes of one k-group of A
                const int usable = a.aregion - 2048;
                // k-groups per chunk: all of them, or (two buffers) an even number that fits half the region
                const int ckg = tkg * rb <= usable ? tkg : (usable / 2 / rb) & ~1;
                const int nch = (tkg + ckg - 1) / ckg;
                for (int m = tid; m < mr; m += FT) {
                    const int loc = locs[m0 + m], li = loc >> 16, lj = loc & 0xffff;
                    rofs[m] = (li * a.stride * a.FW + lj * a.stride) * px;
                }
                __syncthreads();
                for (int c = 0; c < nch; ++c) {
                    const int bs = c & 1;
                    drain(bs);   // the MMAs that read this buffer two chunks ago
                    uint8_t* Ab = Abuf + bs * ckg * rb;
                    const int kg0 = c * ckg, nkg = min(ckg, tkg - kg0);
                    for (int it = tid; it < nkg * mr; it += FT) {
                        const int j = it / mr, m = it - j * mr;
                        const int kg = kg0 + j, prev = kg >= hkg;
                        const int ko = koff[prev ? kg - hkg : kg];
                        uint4 v = make_uint4(0u, 0u, 0u, 0u);
                        if (ko >= 0) {
                            const int e = rofs[m] + ko;
                            if (WP) {
                                const float4* src = reinterpret_cast<const float4*>(R + e);
                                v = pack_bf16x8(src[0], src[1]);
                            } else if (TC_EXACT) {
                                v = *reinterpret_cast<const uint4*>((prev ? Xp : Xt) + e);
                                if (prev) {   // -x_{t-1}: the sign bits of the eight bf16 values, exactly
                                    v.x ^= 0x80008000u;
                                    v.y ^= 0x80008000u;
                                    v.z ^= 0x80008000u;
                                    v.w ^= 0x80008000u;
                                }
                            } else {
                                v = bf16x8_sub(*reinterpret_cast<const uint4*>(Xt + e),
                                               *reinterpret_cast<const uint4*>(Xp + e));
                            }
                        }
                        *reinterpret_cast<uint4*>(Ab + j * rb + m * 16) = v;
                    }
                    fence_proxy_async_smem();
                    ok = __syncthreads_and(ok) != 0;
                    if (!ok) break;
                    if (warp == 0) {
                        tc_fence_after();
                        if (elect_one()) {
                            for (int j = 0; j < nkg; j += 2) {
                                const uint64_t ad = smem_desc(smem_u32(Ab + j * rb), rb, 128, 0);
                                const int wg = kg0 + j < hkg ? kg0 + j : kg0 + j - hkg;   // both halves of A take w
                                const uint64_t bd = smem_desc(smem_u32(Wb + (size_t)wg * SW * 16), SW * 16, 128, 0);
                                mma_bf16(tmem, ad, bd, idesc, (kg0 + j) != 0 ? 1u : 0u);
                            }
                            mma_commit(bs ? bm1 : bm0);
                        }
                        __syncwarp();
                    }
                    pend |= 1u << bs;
                }
                // the last commit covers every MMA issued before it; both buffers' phases advance
                drain(0);
                drain(1);
                ok = __syncthreads_and(ok) != 0;
                if (!ok) break;
                tc_fence_after();
                // D -> shared memory (the A region, free once the MMAs completed), rows SW + 4 floats
                // apart so that the row-per-thread writes spread over the banks; then every thread
                // takes (location, 4 channels) items: z~ += D, y = act(z~ [+ shortcut])
                constexpr int DS = SW + 4;
                float* Dst = reinterpret_cast<float*>(Abuf);
                if (tid < TC_ROWS) {
                    // warp w reads TMEM lanes 32w .. 32w + 31: thread = row = open location m0 + tid,
                    // 32 columns (16 for a 16-channel slice) at a time
                    const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16);
                    constexpr int CC = SW < 32 ? SW : 32;
#pragma unroll 1
                    for (int c0 = 0; c0 < SW; c0 += CC) {
                        uint32_t v[CC];
                        if constexpr (CC == 32) tmem_ld_32x32b_x32(taddr + c0, v);
                        else tmem_ld_32x32b_x16(taddr + c0, v);
                        tmem_wait_ld();
                        if (tid < mr) {
                            float4* drow = reinterpret_cast<float4*>(Dst + tid * DS + c0);
#pragma unroll
                            for (int q = 0; q < CC / 4; ++q)
                                drow[q] = make_float4(__uint_as_float(v[4 * q]), __uint_as_float(v[4 * q + 1]),
                                                      __uint_as_float(v[4 * q + 2]), __uint_as_float(v[4 * q + 3]));
                        }
                    }
                }
                tc_fence_before();
                __syncthreads();
                {
                    const int nq = min(SW, a.Co - o_base) / 4;   // c_out is a multiple of 4
                    for (int it = tid; it < mr * nq; it += FT) {
                        const int m = it / nq, q = it - m * nq;
                        const int loc = locs[m0 + m], li = loc >> 16, lj = loc & 0xffff;
                        const int lz = li * span + lj;
                        const size_t zo = (((size_t)nn * a.Ho + oy0 + li) * a.Wo + ox0 + lj) * a.Co + o_base + 4 * q;
                        const float4 d = reinterpret_cast<const float4*>(Dst + m * DS)[q];
                        const float4 zt = reinterpret_cast<const float4*>(Zs + lz * ZW)[q];
                        float u[4] = {zt.x + d.x, zt.y + d.y, zt.z + d.z, zt.w + d.w};
                        *reinterpret_cast<float4*>(a.z + zo) = make_float4(u[0], u[1], u[2], u[3]);
                        if (y) {
                            const int zi = lz * ZW + 4 * q;
#pragma unroll
                            for (int e = 0; e < 4; ++e) u[e] = activate(has_sc ? u[e] + to_f32(Ss[zi + e]) : u[e], a.act);
                            const __nv_bfloat162 lo = __floats2bfloat162_rn(u[0], u[1]), hi = __floats2bfloat162_rn(u[2], u[3]);
                            uint2 pk;
                            pk.x = *reinterpret_cast<const uint32_t*>(&lo);
                            pk.y = *reinterpret_cast<const uint32_t*>(&hi);
                            *reinterpret_cast<uint2*>(y + zo) = pk;
                        }
                    }
                }
                tc_fence_before();
                __syncthreads();   // D is read before the next pass writes it
            }
            if (!ok) {
                // an MMA never completed (a wait ran out and set the error word): give the ones in
                // flight a last bounded wait before the columns go back
                if (pend & 1u) mbar_wait(bm0, phase & 1u, nullptr, nullptr, LOCAL_WAIT_NS);
                if (pend & 2u) mbar_wait(bm1, (phase >> 1) & 1u, nullptr, nullptr, LOCAL_WAIT_NS);
                __syncthreads();
            }
        }
        if (warp == 0) {
            tc_fence_after();
            tmem_dealloc(tmem, tc_cols<SW>());
        }
    } else {
        constexpr int NQ = SW / 4;
        const int items = (M + FLPI - 1) / FLPI * NQ;
        const int parts = items == 0 ? 1 : max(1, min(8, FT / items));
        auto contract = [&](int item, int k_lo, int k_hi, float (&acc)[FLPI][4], int (&lz)[FLPI]) {
            const int q = item % NQ, mi = item / NQ;
            int rb[FLPI];
#pragma unroll
            for (int u = 0; u < FLPI; ++u) {
                const int m = mi * FLPI + u;
                if (m < M) {
                    const int loc = locs[m], li = loc >> 16, lj = loc & 0xffff;
                    rb[u] = (li * a.stride * a.FW + lj * a.stride) * a.CP;
                    lz[u] = li * span + lj;
                } else {
                    rb[u] = 0;
                    lz[u] = -1;
                }
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[u][j] = 0.f;
            }
            // k = tap * C + ci; walk the taps of [k_lo, k_hi)
            int tap = k_lo / a.C, ci = k_lo - tap * a.C;
            int k = k_lo;
            while (k < k_hi) {
                const int kh = tap / a.KW, kw = tap - (tap / a.KW) * a.KW;
                const int toff = (kh * a.FW + kw) * a.CP;
                const int cend = min(a.C, ci + (k_hi - k));
                const T* wr = Ws + (size_t)(tap * a.C) * SW + q * 4;
#pragma unroll 4
                for (int c = ci; c < cend; ++c) {
                    const float4 w = load_w4(wr + (size_t)c * SW);
#pragma unroll
                    for (int u = 0; u < FLPI; ++u) {
                        const float r = R[rb[u] + toff + c];
                        acc[u][0] = fmaf(r, w.x, acc[u][0]);
                        acc[u][1] = fmaf(r, w.y, acc[u][1]);
                        acc[u][2] = fmaf(r, w.z, acc[u][2]);
                        acc[u][3] = fmaf(r, w.w, acc[u][3]);
                    }
                }
                k += cend - ci;
                ci = 0;
                ++tap;
            }
        };
        auto store = [&](int item, const float (&acc)[FLPI][4], const int (&lz)[FLPI]) {
            const int oq = (item % NQ) * 4;
#pragma unroll
            for (int u = 0; u < FLPI; ++u) {
                if (lz[u] < 0) continue;
                const int li = lz[u] / span, lj = lz[u] - (lz[u] / span) * span;
                const size_t zrow = (((size_t)nn * a.Ho + oy0 + li) * a.Wo + ox0 + lj) * a.Co;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int o = o_base + oq + j;
                    if (o >= a.Co) continue;
                    const int zi = lz[u] * ZW + oq + j;
                    const float znew = Zs[zi] + acc[u][j];
                    a.z[zrow + o] = znew;
                    if (y) y[zrow + o] = y_of(znew, zi);
                }
            }
        };
        if (parts == 1) {
            for (int it = tid; it < items; it += FT) {
                float acc[FLPI][4];
                int lz[FLPI];
                contract(it, 0, a.K, acc, lz);
                store(it, acc, lz);
            }
        } else {
            // too few open locations to occupy the CTA: split k over `parts` thread groups
            const int item = tid % items, part = tid / items;
            float acc[FLPI][4];
            int lz[FLPI];
            if (part < parts) {
                const int k_lo = (int)((long long)a.K * part / parts), k_hi = (int)((long long)a.K * (part + 1) / parts);
                contract(item, k_lo, k_hi, acc, lz);
                if (part > 0) {
#pragma unroll
                    for (int u = 0; u < FLPI; ++u)
#pragma unroll
                        for (int j = 0; j < 4; ++j) red[((part - 1) * items + item) * (FLPI * 4) + u * 4 + j] = acc[u][j];
                }
            }
            __syncthreads();
            if (part == 0) {
                for (int pp = 1; pp < parts; ++pp)
#pragma unroll
                    for (int u = 0; u < FLPI; ++u)
#pragma unroll
                        for (int j = 0; j < 4; ++j) acc[u][j] += red[((pp - 1) * items + item) * (FLPI * 4) + u * 4 + j];
                store(item, acc, lz);
            }
        }
    }

    // with a shortcut: y = act(z + shortcut) at the tile's closed locations (the open ones got theirs above)
    if (y != nullptr && has_sc) {
        const int th = min(span, a.Ho - oy0), tw = min(span, a.Wo - ox0);
        const int nc = DW ? a.Co : min(SW, a.Co - o_base);
        for (int it = tid; it < th * tw * nc; it += FT) {
            const int c = it % nc, p = it / nc;
            const int li = p / tw, lj = p - (p / tw) * tw;
            if (s_open[(li / a.b) * a.sb + lj / a.b]) continue;
            const int zi = (li * span + lj) * zw + c;
            y[(((size_t)nn * a.Ho + oy0 + li) * a.Wo + ox0 + lj) * a.Co + o_base + c] = y_of(Zs[zi], zi);
        }
    }
    if (sl == 0 && warp == 0 && list_bal) {
        const int basei = __shfl_sync(0xffffffffu, list_base, 0);
        if (list_open) {
            const int by = ty * a.sb + lane / a.sb, bx = tx * a.sb + lane % a.sb;
            a.list[basei + __popc(list_bal & ((1u << lane) - 1u))] = (int32_t)(((size_t)nn * a.nby + by) * a.nbx + bx);
        }
    }
}

// Weights of the staged form, in the layer's dtype: dense [slice][K][sw]
// (K index = tap * c_in + ci, channels past c_out zero), depthwise [taps][C].
template <typename T>
__global__ void pack_local_weights_kernel(const float* __restrict__ wcc, T* __restrict__ out, int K, int Co,
                                          int nsl, int sw, int dw)
{
    const long long total = dw ? (long long)K * Co : (long long)nsl * K * sw;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        if (dw) {
            out[i] = from_f32<T>(wcc[i]);
        } else {
            const int j = (int)(i % sw);
            const long long rest = i / sw;
            const int k = (int)(rest % K), sl = (int)(rest / K);
            const int o = sl * sw + j;
            out[i] = from_f32<T>(o < Co ? wcc[(size_t)k * Co + o] : 0.f);
        }
    }
}

// Weights of the tensor-core contraction: per slice, [Kp/8][sw][8] bf16 (the
// no-swizzle K-major layout of the MMA's B operand), element (k, n) = w(k, o)
// with o = slice * sw + n, k = tap * c_in + ci; zero for k >= K and o >= c_out.
__global__ void pack_local_tc_weights_kernel(const float* __restrict__ wcc, __nv_bfloat16* __restrict__ out, int K,
                                             int Kp, int Co, int nsl, int sw)
{
    const long long total = (long long)nsl * Kp * sw;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int e = (int)(i % 8);
        long long rest = i / 8;
        const int n = (int)(rest % sw);
        rest /= sw;
        const int g = (int)(rest % (Kp / 8)), sl = (int)(rest / (Kp / 8));
        const int k = g * 8 + e, o = sl * sw + n;
        out[i] = __float2bfloat16_rn(o < Co && k < K ? wcc[(size_t)k * Co + o] : 0.f);
    }
}

struct LocalShape {
    int sb, span, FH, FW, CP;
    size_t smem;
};

LocalShape local_shape(const Layer& L, int sb)
{
    LocalShape s;
    s.sb = sb;
    s.span = sb * L.p.block;
    s.FH = (s.span - 1) * L.p.stride + L.p.k_h;
    s.FW = (s.span - 1) * L.p.stride + L.p.k_w;
    s.CP = L.p.c_in | 1;   // odd pixel stride: neighbouring locations fall in different banks
    const size_t fp = (size_t)s.FH * s.FW;
    // residual, norms, location table, and the dense contraction's weight chunk and offsets
    s.smem = (fp * s.CP + fp + (size_t)s.span * s.span + 3 + (size_t)GKC * L.p.c_out + GKC) * sizeof(float);
    return s;
}

LocalShape choose_shape(const Layer& L)
{
    int sb = L.p.block >= 4 ? 1 : (4 + L.p.block - 1) / L.p.block;
    LocalShape s = local_shape(L, sb);
    while (s.smem > LOCAL_MAX_SMEM && sb > 1) s = local_shape(L, --sb);
    return s;
}

template <typename T>
const void* kernel_of(const Layer& L)
{
    if (L.cpg == 1 && L.opg == 1) return (const void*)step_local_kernel<T, true, false>;
    if (L.p.c_out % 4 == 0 && L.opg % 4 == 0) return (const void*)step_local_kernel<T, false, true>;
    return (const void*)step_local_kernel<T, false, false>;
}

const void* kernel_of(const Layer& L)
{
    return L.p.dtype == SKIPCONV_BF16 ? kernel_of<__nv_bfloat16>(L) : kernel_of<float>(L);
}

// ------------------------------------------------------ staged form, host side
struct StagedShape {
    LocalShape g;
    int sw;          // output channels per CTA (dense layers)
    int nsl;
    int zw;          // channels of the z / shortcut tile boxes
    int Kp;          // tensor-core contraction: K rounded up to 16 (else K)
    size_t own_max;  // most input pixels a tile owns
    uint32_t wbytes;
    uint32_t off_xp, off_w, off_r, off_p, off_loc, off_scr, off_z, off_sc, off_chg, off_dq, off_a;
    int aregion;     // tensor-core contraction: bytes for A (all of it in one go where that fits)
    size_t smem;
};

inline uint32_t up128(size_t v) { return (uint32_t)((v + 127) & ~(size_t)127); }

bool is_depthwise(const Layer& L) { return L.cpg == 1 && L.opg == 1; }

StagedShape staged_shape(const Layer& L, int sb, bool wp = false)
{
    StagedShape t;
    t.g = local_shape(L, sb);
    t.g.CP = L.p.c_in + 4;   // 16-byte aligned residual rows, consecutive pixels 4 banks apart
    const bool dw = is_depthwise(L);
    const size_t fp = (size_t)t.g.FH * t.g.FW;
    const int K = L.p.k_h * L.p.k_w * L.p.c_in;
    const bool tc = L.local_tc && !dw;
    // small tiles with few output channels: narrower slices spread an open tile over more SMs.  A
    // kernel that uses the tensor cores runs one CTA per SM (the occupancy the runtime reports for a
    // kernel with tcgen05 instructions), so there a slice is always 32 channels wide: half the CTAs
    // of 16-channel slices (c2: 120-121 against 125 us per frame), while 64- and 128-channel
    // slices were slower (129 us; c3 123 against 107 us)
    t.sw = tc ? SW_WIDE : (t.g.span <= 4 && L.p.c_out <= 32) ? SW_NARROW : SW_WIDE;
    t.nsl = dw ? 1 : (L.p.c_out + t.sw - 1) / t.sw;
    t.zw = dw ? L.p.c_out : t.sw;
    // the tensor-core contraction's weights: [K/8][sw][8] bf16, K padded to the MMA's K step
    t.Kp = tc ? (K + 15) / 16 * 16 : K;
    const size_t wb = dw ? (size_t)L.p.k_h * L.p.k_w * L.p.c_in * L.esize : (size_t)t.Kp * t.sw * L.esize;
    t.wbytes = (uint32_t)((wb + 15) & ~(size_t)15);
    // largest owned input region of a tile (the last tile row / column owns the rest of the frame)
    const int span_in = t.g.span * L.p.stride;
    const int nty = (L.nby + sb - 1) / sb, ntx = (L.nbx + sb - 1) / sb;
    const int own_h = std::max(std::min(span_in, L.p.h), L.p.h - (nty - 1) * span_in);
    const int own_w = std::max(std::min(span_in, L.p.w), L.p.w - (ntx - 1) * span_in);
    t.own_max = (size_t)std::max(own_h, 0) * std::max(own_w, 0);
    const size_t tile_elems = (size_t)t.g.span * t.g.span * t.zw;
    const uint32_t xb = up128(fp * L.p.c_in * L.esize);
    // the previous input's footprint: x_{t-1} in the dtype, or (wp) its warp T(x_{t-1}) in fp32
    const uint32_t pb = wp ? up128(fp * L.p.c_in * sizeof(float)) : xb;
    t.off_xp = xb;
    t.off_w = xb + pb;
    t.off_r = t.off_w + up128(t.wbytes);
    // the fp32 residual: the FMA contraction's and the warped tensor-core step's operand
    t.off_p = t.off_r + ((dw || (tc && !wp)) ? 0 : up128(fp * t.g.CP * sizeof(float)));
    t.off_loc = t.off_p + up128(fp * sizeof(float));
    t.off_scr = t.off_loc + up128((size_t)t.g.span * t.g.span * sizeof(int));
    // scratch: the footprint pass's chunk partials, later (dense) the k-split partial sums
    const size_t chunks = fp * (L.p.c_in * L.esize / 16);
    // (the tensor-core contraction keeps its k-group and row offset tables there instead)
    const size_t scr = std::max(chunks * (sizeof(float) + 1),
                                dw ? (size_t)0
                                   : tc ? (size_t)(TC_MAX_KG + TC_ROWS) * sizeof(int)
                                        : (size_t)FT * FLPI * 4 * sizeof(float));
    t.off_z = t.off_scr + up128(scr);
    t.off_sc = t.off_z + up128(tile_elems * sizeof(float));
    t.off_chg = t.off_sc + (L.p.emit_y ? up128(tile_elems * L.esize) : 0);
    t.off_dq = t.off_chg + up128(t.own_max);
    t.off_a = t.off_dq + up128(fp);
    // A for a whole pass of the tile's locations (at most 128 rows) in one go, plus the 2 KB an MMA may
    // read past it, where that fits TC_AREGION_MAX; else TC_AREGION_MAX, built in chunks
    const size_t a_rows = (size_t)std::min(128, t.g.span * t.g.span);
    const size_t a_kg = (size_t)(t.Kp / 8) * ((TC_EXACT && !wp) ? 2 : 1);
    const size_t a_need = a_kg * ((a_rows + 7) / 8 * 8) * 16 + 2048;
    const size_t d_need = ((a_rows + 7) / 8 * 8) * (size_t)(t.sw + 4) * sizeof(float);   // D staged for the epilogue
    t.aregion = tc ? (int)up128(std::max(std::min(a_need, (size_t)TC_AREGION_MAX), d_need)) : 0;
    t.smem = (size_t)t.off_a + t.aregion + 1024;
    return t;
}

// The staged form needs TMA boxes of the footprint (a pixel's channels a
// multiple of 16 bytes, every box edge at most 256), of the z tile (c_out a
// multiple of 4) and of the shortcut tile (c_out a multiple of 16 bytes of
// the dtype), and a dense (groups = 1) or depthwise layer.
bool staged_ok(const Layer& L, StagedShape* out, bool wp = false)
{
    if (!(L.p.groups == 1 || is_depthwise(L))) return false;
    if ((L.p.c_in * L.esize) % 16 || L.p.c_in > 256) return false;
    if (L.p.c_out % 4 || (L.p.emit_y && (L.p.c_out * L.esize) % 16)) return false;
    int sb = L.p.block >= 4 ? 1 : (4 + L.p.block - 1) / L.p.block;
    StagedShape t = staged_shape(L, sb, wp);
    while (t.smem > LOCAL_MAX_SMEM && sb > 1) t = staged_shape(L, --sb, wp);
    if (t.smem > LOCAL_MAX_SMEM || t.g.FH > 256 || t.g.FW > 256 || t.g.span > 256 || t.zw > 256) return false;
    if ((long long)L.p.n_streams * ((L.nby + sb - 1) / sb) * ((L.nbx + sb - 1) / sb) * t.nsl > 0x7fffffffLL)
        return false;
    if (out) *out = t;
    return true;
}

bool encode_footprint_map(CUtensorMap* m, const void* base, const Layer& L, const StagedShape& t)
{
    EncodeTiledFn enc = encode_tiled_fn();
    if (!enc) return false;
    const cuuint64_t C = L.p.c_in, W = L.p.w, H = L.p.h, N = L.p.n_streams, es = L.esize;
    cuuint64_t dims[4] = {C, W, H, N};
    cuuint64_t strides[3] = {C * es, W * C * es, H * W * C * es};
    cuuint32_t box[4] = {(cuuint32_t)C, (cuuint32_t)t.g.FW, (cuuint32_t)t.g.FH, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUtensorMapDataType dt =
        L.p.dtype == SKIPCONV_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    return enc(m, dt, 4, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tile boxes of an output-shaped tensor [n][ho][wo][c_out]: z (fp32) or the shortcut (dtype).
bool encode_tile_map(CUtensorMap* m, const void* base, const Layer& L, const StagedShape& t, bool fp32)
{
    EncodeTiledFn enc = encode_tiled_fn();
    if (!enc) return false;
    const cuuint64_t Co = L.p.c_out, Wo = L.wo, Ho = L.ho, N = L.p.n_streams, es = fp32 ? 4 : L.esize;
    cuuint64_t dims[4] = {Co, Wo, Ho, N};
    cuuint64_t strides[3] = {Co * es, Wo * Co * es, Ho * Wo * Co * es};
    cuuint32_t box[4] = {(cuuint32_t)t.zw, (cuuint32_t)t.g.span, (cuuint32_t)t.g.span, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUtensorMapDataType dt = fp32 || L.p.dtype != SKIPCONV_BF16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32
                                                                     : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    return enc(m, dt, 4, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <typename T, bool WP>
const void* staged_kernel_of(const Layer& L, int sw)
{
    if (is_depthwise(L)) return (const void*)step_local_staged_kernel<T, true, SW_WIDE, WP, false>;
    return sw == SW_NARROW ? (const void*)step_local_staged_kernel<T, false, SW_NARROW, WP, false>
                           : (const void*)step_local_staged_kernel<T, false, SW_WIDE, WP, false>;
}

template <bool WP>
const void* staged_tc_kernel_of(int)
{
    return (const void*)step_local_staged_kernel<__nv_bfloat16, false, SW_WIDE, WP, true>;
}

const void* staged_kernel_of(const Layer& L, int sw, bool wp = false)
{
    if (L.p.dtype == SKIPCONV_BF16) {
        if (L.local_tc) return wp ? staged_tc_kernel_of<true>(sw) : staged_tc_kernel_of<false>(sw);
        return wp ? staged_kernel_of<__nv_bfloat16, true>(L, sw) : staged_kernel_of<__nv_bfloat16, false>(L, sw);
    }
    return wp ? staged_kernel_of<float, true>(L, sw) : staged_kernel_of<float, false>(L, sw);
}

// The staged form's warped variant runs where it tiles the frame, slices the
// channels and packs the weights as the plain form does (the z tile map, the
// per-tile flags and the packed weights are the plain form's).
bool staged_wp_ok(const Layer& L, StagedShape* t, StagedShape* tw)
{
    if (!L.local_staged || !staged_ok(L, t) || !staged_ok(L, tw, true)) return false;
    return tw->g.sb == t->g.sb && tw->g.span == t->g.span && tw->g.FH == t->g.FH && tw->g.FW == t->g.FW &&
           tw->zw == t->zw && tw->sw == t->sw && tw->nsl == t->nsl && tw->wbytes == t->wbytes;
}

// Warped residual (Eq. 10-11), before the step, in one pass over the frame with
// the bilinear weights taken once per pixel:
//   - the output state's warp z~ <- T~(z~_{t-1}) from zsrc into zdst (the layer
//     keeps the frame size, so T~ uses the same flow), and y = act of it when y
//     is given (a step without a shortcut refreshes y only at open blocks);
//   - for the staged form (tx != NULL), T(x_{t-1}) into an fp32 frame, and the
//     commit of x_t with the pixels' change flags, which compare the raw frames.
// A group of 2^lp_log2 lanes per pixel, 16-byte vectors of channels.
struct WarpPreArgs {
    const float* flow;
    const float* zsrc;
    float* zdst;
    void* y;
    const void* xt;
    const void* xp;
    void* xn;
    const uint8_t* chg_prev;
    uint8_t* chg_cur;
    float* tx;
    int n, H, W, C, Co, act, lp_log2;
};

__device__ __forceinline__ void unpack16(const uint4& v, float (&f)[8], const float*)
{
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y); f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
}
__device__ __forceinline__ void unpack16(const uint4& v, float (&f)[8], const __nv_bfloat16*)
{
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 t = __bfloat1622float2(h[k]);
        f[2 * k] = t.x;
        f[2 * k + 1] = t.y;
    }
}
__device__ __forceinline__ void store_act4(float* y, const float4& v, int act)
{
    *reinterpret_cast<float4*>(y) = make_float4(activate(v.x, act), activate(v.y, act), activate(v.z, act), activate(v.w, act));
}
__device__ __forceinline__ void store_act4(__nv_bfloat16* y, const float4& v, int act)
{
    __nv_bfloat162 h[2] = {__floats2bfloat162_rn(activate(v.x, act), activate(v.y, act)),
                           __floats2bfloat162_rn(activate(v.z, act), activate(v.w, act))};
    *reinterpret_cast<uint2*>(y) = *reinterpret_cast<const uint2*>(h);
}

template <typename T>
__global__ void __launch_bounds__(256) warp_pre_kernel(const WarpPreArgs a)
{
    constexpr int VX = 16 / (int)sizeof(T);
    const int LP = 1 << a.lp_log2;
    const int g = threadIdx.x & (LP - 1);
    const long long npx = (long long)a.n * a.H * a.W;
    const long long ngroups = ((long long)gridDim.x * blockDim.x) >> a.lp_log2;
    // the lanes of a warp iterate together (the change flag is a shuffle reduction over each group)
    const long long gid = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> a.lp_log2;
    const long long gid0 = gid - ((threadIdx.x & 31) >> a.lp_log2);
    const T* xt = static_cast<const T*>(a.xt);
    const T* xp = static_cast<const T*>(a.xp);
    T* xn = static_cast<T*>(a.xn);
    T* y = static_cast<T*>(a.y);
    for (long long it = 0; gid0 + it < npx; it += ngroups) {
        const long long p = gid + it;
        const bool live = p < npx;
        Bilinear bl = {};
        if (live) {
            const int ix = (int)(p % a.W), iy = (int)((p / a.W) % a.H), nn = (int)(p / ((long long)a.W * a.H));
            bl = bilinear_of(a.flow, nn, a.H, a.W, 1, iy, ix);   // offsets in pixels
        }
        if (a.tx) {
            unsigned d = 0;
            if (live) {
                for (int k = g; k < a.C / VX; k += LP) {
                    const size_t e = (size_t)p * a.C + (size_t)k * VX;
                    const uint4 av = *reinterpret_cast<const uint4*>(xt + e);
                    const uint4 bv = *reinterpret_cast<const uint4*>(xp + e);
                    d |= (av.x ^ bv.x) | (av.y ^ bv.y) | (av.z ^ bv.z) | (av.w ^ bv.w);
                    float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        float f[8];
                        unpack16(*reinterpret_cast<const uint4*>(xp + bl.off[q] * a.C + (size_t)k * VX), f, (const T*)nullptr);
#pragma unroll
                        for (int j = 0; j < VX; ++j) v[j] += bl.wt[q] * f[j];
                    }
                    float4* o = reinterpret_cast<float4*>(a.tx + e);
                    o[0] = make_float4(v[0], v[1], v[2], v[3]);
                    if (VX == 8) o[1] = make_float4(v[4], v[5], v[6], v[7]);
                }
            }
            for (int o = LP >> 1; o > 0; o >>= 1) d |= __shfl_xor_sync(0xffffffffu, d, o);
            if (live) {
                const bool changed = d != 0;
                if (changed || a.chg_prev[p])
                    for (int k = g; k < a.C / VX; k += LP) {
                        const size_t e = (size_t)p * a.C + (size_t)k * VX;
                        *reinterpret_cast<uint4*>(xn + e) = *reinterpret_cast<const uint4*>(xt + e);
                    }
                if (g == 0) a.chg_cur[p] = changed ? 1 : 0;
            }
        }
        if (!live) continue;
        if ((a.Co & 3) == 0) {
            for (int k = g; k < a.Co / 4; k += LP) {
                float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float4 zq = *reinterpret_cast<const float4*>(a.zsrc + bl.off[q] * a.Co + (size_t)k * 4);
                    v.x += bl.wt[q] * zq.x;
                    v.y += bl.wt[q] * zq.y;
                    v.z += bl.wt[q] * zq.z;
                    v.w += bl.wt[q] * zq.w;
                }
                const size_t e = (size_t)p * a.Co + (size_t)k * 4;
                *reinterpret_cast<float4*>(a.zdst + e) = v;
                if (y) store_act4(y + e, v, a.act);
            }
        } else {
            for (int c = g; c < a.Co; c += LP) {
                float v = 0.f;
#pragma unroll
                for (int q = 0; q < 4; ++q) v += bl.wt[q] * a.zsrc[bl.off[q] * a.Co + c];
                const size_t e = (size_t)p * a.Co + c;
                a.zdst[e] = v;
                if (y) y[e] = from_f32<T>(activate(v, a.act));
            }
        }
    }
}

cudaLaunchConfig_t pdl_config(const Layer& L, long long grid, int threads, size_t smem, cudaLaunchAttribute* attr)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = L.stream;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cfg;
}

// The staged form's launch: tm_prev maps the previous input's footprints (x_{t-1}; for a warped
// step T(x_{t-1}) in fp32, wp = true).
// CTAs of a staged-form launch resident on the GPU at once, from the SM's register file, shared
// memory and thread slots (the static limits).  The runtime's occupancy query answers one CTA per SM
// for the instantiations that contain tcgen05 instructions whatever their size, while the SMs run
// two or three of them (the limits ncu reports, and the start times of their CTAs).
cudaError_t staged_resident(const Layer& L, const void* kernel, size_t smem, int* resident)
{
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, kernel);
    int regs_sm = 0, smem_sm = 0, smem_reserved = 0, threads_sm = 0;
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, L.device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, L.device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&smem_reserved, cudaDevAttrReservedSharedMemoryPerBlock, L.device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&threads_sm, cudaDevAttrMaxThreadsPerMultiProcessor, L.device);
    if (e != cudaSuccess) return e;
    // registers are allocated per warp in units of 256
    const int warp_regs = (fa.numRegs * 32 + 255) / 256 * 256;
    const int by_regs = regs_sm / (warp_regs * (FT / 32));
    const int by_smem = smem_sm / (int)(smem + fa.sharedSizeBytes + smem_reserved);
    const int by_threads = threads_sm / FT;
    const int per_sm = std::max(1, std::min(by_regs, std::min(by_smem, by_threads)));
    *resident = L.num_sms * per_sm;
    return cudaSuccess;
}

cudaError_t launch_staged(Layer& L, const StagedShape& t, const void* x_t, const void* shortcut, int force,
                          const Layer* px, const Layer* psc, const CUtensorMap* tm_prev, bool wp)
{
    const int cur = (int)(L.t & 1), nxt = cur ^ 1;
    cudaLaunchAttribute attr[1];
    alignas(64) CUtensorMap tm_xt;
    if (!encode_footprint_map(&tm_xt, x_t, L, t)) {
        set_error("tensor map of x_t rejected");
        return cudaErrorInvalidValue;
    }
    FastArgs a;
    a.wpack = L.w_loc;
    a.wbytes = t.wbytes;
    a.xt = x_t;
    a.xp = L.xbuf[cur];
    a.xn = L.xbuf[nxt];
    a.chg_prev = L.chg[nxt];
    a.chg_cur = L.chg[cur];
    a.z = L.z;
    a.y = L.y;
    a.sc = L.y ? shortcut : nullptr;
    a.mask = L.mask;
    a.list = L.list;
    a.count_cur = step_count(L);
    a.count_next = next_count(L);
    a.err = L.err_dev;
    a.force = force;
    a.n = L.p.n_streams; a.H = L.p.h; a.W = L.p.w; a.C = L.p.c_in; a.Ho = L.ho; a.Wo = L.wo;
    a.Co = L.p.c_out; a.KH = L.p.k_h; a.KW = L.p.k_w; a.stride = L.p.stride; a.pad = L.p.pad; a.b = L.p.block;
    a.nby = L.nby; a.nbx = L.nbx; a.act = L.p.activation;
    a.sb = t.g.sb;
    a.nty = (L.nby + t.g.sb - 1) / t.g.sb;
    a.ntx = (L.nbx + t.g.sb - 1) / t.g.sb;
    a.FH = t.g.FH; a.FW = t.g.FW; a.CP = t.g.CP; a.nsl = t.nsl; a.K = L.p.k_h * L.p.k_w * L.p.c_in;
    a.Kp = t.Kp;
    a.off_xp = t.off_xp; a.off_w = t.off_w; a.off_r = t.off_r; a.off_p = t.off_p; a.off_loc = t.off_loc;
    a.off_scr = t.off_scr; a.off_z = t.off_z; a.off_sc = t.off_sc; a.off_chg = t.off_chg; a.off_dq = t.off_dq;
    a.off_a = t.off_a;
    a.aregion = t.aregion;
    a.thr = L.gate_thr;
    a.px_chg = px ? px->ychg : nullptr;
    a.pxb = px ? px->p.block : 1; a.pxnby = px ? px->nby : 1; a.pxnbx = px ? px->nbx : 1;
    a.psc_chg = psc ? psc->ychg : nullptr;
    a.pscb = psc ? psc->p.block : 1; a.pscnby = psc ? psc->nby : 1; a.pscnbx = psc ? psc->nbx : 1;
    a.ychg = L.ychg;
    a.tile_chg_prev = L.tile_chg + (size_t)nxt * L.ntiles;
    a.tile_chg_cur = L.tile_chg + (size_t)cur * L.ntiles;
    alignas(64) CUtensorMap tm_sc = L.tmap_ztile;   // unused without a shortcut
    if (a.sc && !encode_tile_map(&tm_sc, a.sc, L, t, false)) {
        set_error("tensor map of the shortcut rejected");
        return cudaErrorInvalidValue;
    }
    const long long grid = (long long)a.n * a.nty * a.ntx * t.nsl;
    cudaLaunchConfig_t cfg = pdl_config(L, grid, FT, t.smem, attr);
    CUtensorMap* tm_z = const_cast<CUtensorMap*>(&L.tmap_ztile);
    void* args[] = {&tm_xt, const_cast<CUtensorMap*>(tm_prev), tm_z, &tm_sc, &a};
    return cudaLaunchKernelExC(&cfg, staged_kernel_of(L, t.sw, wp), args);
}

}  // namespace

bool step_local_preferred(const Layer& L)
{
    if (L.p.gate == SKIPCONV_GATE_GUMBEL || L.p.dense_mode) return false;
    const double dense_macs = (double)L.p.n_streams * L.ho * L.wo * L.p.c_out * L.cpg * L.p.k_h * L.p.k_w;
    return dense_macs <= LOCAL_AUTO_MAX_MACS && staged_ok(L, nullptr);
}

bool step_local_warp_supported(const Layer& L)
{
    return L.fused == 2 && L.p.stride == 1 && L.ho == L.p.h && L.wo == L.p.w &&
           choose_shape(L).smem <= LOCAL_MAX_SMEM;
}

bool step_local_supported(const Layer& L)
{
    if (L.path != SKIPCONV_PATH_CUDA_CORE || L.p.conv_path == SKIPCONV_PATH_CUDA_CORE_SEPARATE) return false;
    if (L.p.gate == SKIPCONV_GATE_GUMBEL) return false;
    return staged_ok(L, nullptr) || choose_shape(L).smem <= LOCAL_MAX_SMEM;
}

// Layers that keep y publish, per gate block, whether a step may have changed it
// (read by linked consumers).  All ones until the first step (a key frame).
static cudaError_t alloc_ychg(Layer& L)
{
    if (!L.y) return cudaSuccess;
    const size_t nblk = (size_t)L.p.n_streams * L.nby * L.nbx;
    cudaError_t e = cudaMalloc((void**)&L.ychg, nblk);
    if (e != cudaSuccess) {
        L.ychg = nullptr;
        return e;
    }
    L.state_bytes += nblk;
    return cudaMemsetAsync(L.ychg, 1, nblk, L.stream);
}

cudaError_t step_local_prepare(Layer& L)
{
    StagedShape t;
    // the tensor-core contraction needs the staged form (and room for its A region), and its k-group
    // offset table holds TC_MAX_KG entries
    if (L.local_tc && (L.p.dtype != SKIPCONV_BF16 || is_depthwise(L) || L.p.groups != 1 ||
                       (L.p.k_h * L.p.k_w * L.p.c_in + 15) / 16 * 2 > TC_MAX_KG || !staged_ok(L, nullptr)))
        L.local_tc = 0;
    if (staged_ok(L, &t)) {
        if (!encode_footprint_map(&L.tmap_fp[0], L.xbuf[0], L, t) || !encode_footprint_map(&L.tmap_fp[1], L.xbuf[1], L, t) ||
            !encode_tile_map(&L.tmap_ztile, L.z, L, t, true)) {
            set_error("tensor map of the layer state rejected");
            return cudaErrorInvalidValue;
        }
        const size_t bytes = (size_t)t.wbytes * t.nsl;
        cudaError_t e = cudaMalloc(&L.w_loc, bytes);
        if (e != cudaSuccess) {
            L.w_loc = nullptr;
            return e;
        }
        L.state_bytes += bytes;
        e = cudaMemsetAsync(L.w_loc, 0, bytes, L.stream);
        if (e != cudaSuccess) return e;
        const bool dw = is_depthwise(L);
        const int K = L.p.k_h * L.p.k_w * L.p.c_in;
        const long long total = dw ? (long long)K * L.p.c_out : (long long)t.nsl * t.Kp * t.sw;
        const int grid = (int)((total + 255) / 256 < 4096 ? (total + 255) / 256 : 4096);
        if (L.local_tc)
            pack_local_tc_weights_kernel<<<grid, 256, 0, L.stream>>>(L.w_cc, (__nv_bfloat16*)L.w_loc, K, t.Kp,
                                                                     L.p.c_out, t.nsl, t.sw);
        else if (L.p.dtype == SKIPCONV_BF16)
            pack_local_weights_kernel<__nv_bfloat16><<<grid, 256, 0, L.stream>>>(
                L.w_cc, (__nv_bfloat16*)L.w_loc, dw ? L.p.k_h * L.p.k_w : K, L.p.c_out, t.nsl, t.sw, dw ? 1 : 0);
        else
            pack_local_weights_kernel<float><<<grid, 256, 0, L.stream>>>(L.w_cc, (float*)L.w_loc,
                                                                         dw ? L.p.k_h * L.p.k_w : K, L.p.c_out,
                                                                         t.nsl, t.sw, dw ? 1 : 0);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        L.local_staged = 1;
        L.ntiles = (int)((long long)L.p.n_streams * ((L.nby + t.g.sb - 1) / t.g.sb) * ((L.nbx + t.g.sb - 1) / t.g.sb));
        e = cudaMalloc((void**)&L.tile_chg, 2 * (size_t)L.ntiles);
        if (e != cudaSuccess) {
            L.tile_chg = nullptr;
            return e;
        }
        L.state_bytes += 2 * (size_t)L.ntiles;
        e = cudaMemsetAsync(L.tile_chg, 0, 2 * (size_t)L.ntiles, L.stream);
        if (e == cudaSuccess) e = alloc_ychg(L);
        if (e == cudaSuccess) e = ensure_dynamic_smem(staged_kernel_of(L, t.sw), t.smem);
        if (e == cudaSuccess) e = staged_resident(L, staged_kernel_of(L, t.sw), t.smem, &L.local_resident);
        // warped steps run the staged form's warped variant, or the general form when it does not fit
        StagedShape tp, tw;
        if (e == cudaSuccess && staged_wp_ok(L, &tp, &tw)) e = ensure_dynamic_smem(staged_kernel_of(L, tw.sw, true), tw.smem);
        if (e == cudaSuccess && choose_shape(L).smem <= LOCAL_MAX_SMEM) e = ensure_dynamic_smem(kernel_of(L), choose_shape(L).smem);
        return e;
    }
    L.local_staged = 0;
    const cudaError_t e = alloc_ychg(L);
    if (e != cudaSuccess) return e;
    return ensure_dynamic_smem(kernel_of(L), choose_shape(L).smem);
}

cudaError_t launch_step_warp_pass(Layer& L, const void* x_t, const void* shortcut, const float* flow)
{
    const int cur = (int)(L.t & 1), nxt = cur ^ 1;
    StagedShape t, tw;
    const bool staged = staged_wp_ok(L, &t, &tw);
    const size_t nz = (size_t)L.p.n_streams * L.ho * L.wo * L.p.c_out;
    const size_t nx = (size_t)L.p.n_streams * L.p.h * L.p.w * L.p.c_in;
    cudaError_t e = cudaSuccess;
    if (!L.z_prev) {
        e = cudaMalloc((void**)&L.z_prev, nz * sizeof(float));
        if (e != cudaSuccess) {
            L.z_prev = nullptr;
            return e;
        }
        L.state_bytes += nz * sizeof(float);
    }
    if (staged && !L.tx) {
        e = cudaMalloc((void**)&L.tx, nx * sizeof(float));
        if (e != cudaSuccess) {
            L.tx = nullptr;
            return e;
        }
        L.state_bytes += nx * sizeof(float);
        EncodeTiledFn enc = encode_tiled_fn();
        const cuuint64_t C = L.p.c_in, W = L.p.w, H = L.p.h, N = L.p.n_streams;
        cuuint64_t dims[4] = {C, W, H, N};
        cuuint64_t strides[3] = {C * 4, W * C * 4, H * W * C * 4};
        cuuint32_t box[4] = {(cuuint32_t)C, (cuuint32_t)tw.g.FW, (cuuint32_t)tw.g.FH, 1};
        cuuint32_t estr[4] = {1, 1, 1, 1};
        if (!enc || enc(&L.tmap_tx, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, L.tx, dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
            set_error("tensor map of the warped frame rejected");
            return cudaErrorInvalidValue;
        }
    }
    WarpPreArgs w;
    w.flow = flow;
    w.zsrc = L.z;
    w.zdst = L.z_prev;
    w.y = L.y && !shortcut ? L.y : nullptr;
    w.xt = x_t;
    w.xp = L.xbuf[cur];
    w.xn = L.xbuf[nxt];
    w.chg_prev = L.chg[nxt];
    w.chg_cur = L.chg[cur];
    w.tx = staged ? L.tx : nullptr;
    w.n = L.p.n_streams; w.H = L.p.h; w.W = L.p.w; w.C = L.p.c_in; w.Co = L.p.c_out; w.act = L.p.activation;
    const int vx = 16 / L.esize;
    int chunks = (L.p.c_out % 4 == 0) ? L.p.c_out / 4 : L.p.c_out;
    if (staged) chunks = std::max(chunks, L.p.c_in / vx);
    w.lp_log2 = 0;
    while ((1 << w.lp_log2) < chunks && w.lp_log2 < 5) ++w.lp_log2;
    const long long npx = (long long)L.p.n_streams * L.p.h * L.p.w;
    const long long per_block = 256 >> w.lp_log2;
    const long long blocks = (npx + per_block - 1) / per_block, cap = (long long)L.num_sms * 8;
    const int grid = (int)(blocks < cap ? blocks : cap);
    if (L.p.dtype == SKIPCONV_BF16) warp_pre_kernel<__nv_bfloat16><<<grid, 256, 0, L.stream>>>(w);
    else warp_pre_kernel<float><<<grid, 256, 0, L.stream>>>(w);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    std::swap(L.z, L.z_prev);
    if (L.local_staged && !encode_tile_map(&L.tmap_ztile, L.z, L, t, true)) {
        set_error("tensor map of the layer state rejected");
        return cudaErrorInvalidValue;
    }
    return cudaSuccess;
}

cudaError_t launch_step_local(Layer& L, const void* x_t, const void* shortcut, int force, const Layer* px,
                              const Layer* psc, const float* flow)
{
    const int cur = (int)(L.t & 1), nxt = cur ^ 1;
    cudaLaunchAttribute attr[1];
    StagedShape t;
    StagedShape tw;
    if (flow && staged_wp_ok(L, &t, &tw))
        return launch_staged(L, tw, x_t, shortcut, force, nullptr, nullptr, &L.tmap_tx, true);
    if (L.local_staged && !flow) {
        if (!staged_ok(L, &t)) return cudaErrorInvalidValue;
        // Linked inputs pay only where the grid is several waves of resident CTAs: skipped tiles then
        // take whole waves off the step.  Within one or two waves the step lasts about as long as its
        // slowest (open) tiles, and the flag read would only delay each tile's footprint load by a
        // memory round trip (measured: c2 linked 137.7 against 125.2 us unlinked at 1.26 waves); such
        // a step reads the whole frame instead.
        if ((long long)L.ntiles * t.nsl <= 2LL * L.local_resident) px = psc = nullptr;
        return launch_staged(L, t, x_t, shortcut, force, px, psc, &L.tmap_fp[cur], false);
    }
    const LocalShape s = choose_shape(L);
    LocalArgs a;
    a.xt = x_t;
    a.xp = L.xbuf[cur];
    a.xn = L.xbuf[nxt];
    a.chg_prev = L.chg[nxt];
    a.chg_cur = L.chg[cur];
    a.wcc = L.w_cc;
    a.z = L.z;
    a.y = L.y;
    a.sc = L.y ? shortcut : nullptr;
    a.mask = L.mask;
    a.list = L.list;
    a.count_cur = step_count(L);
    a.count_next = next_count(L);
    a.force = force;
    a.n = L.p.n_streams; a.H = L.p.h; a.W = L.p.w; a.C = L.p.c_in; a.Ho = L.ho; a.Wo = L.wo; a.Co = L.p.c_out;
    a.KH = L.p.k_h; a.KW = L.p.k_w; a.stride = L.p.stride; a.pad = L.p.pad; a.b = L.p.block;
    a.nby = L.nby; a.nbx = L.nbx; a.cpg = L.cpg; a.opg = L.opg; a.groups = L.p.groups; a.act = L.p.activation;
    a.sb = s.sb;
    a.nty = (L.nby + s.sb - 1) / s.sb;
    a.ntx = (L.nbx + s.sb - 1) / s.sb;
    a.FH = s.FH; a.FW = s.FW; a.CP = s.CP;
    a.thr = L.gate_thr;
    a.ychg = L.ychg;
    a.psc_chg = psc ? psc->ychg : nullptr;
    a.pscb = psc ? psc->p.block : 1; a.pscnby = psc ? psc->nby : 1; a.pscnbx = psc ? psc->nbx : 1;
    a.flow = flow;
    (void)px;   // the general form reads every tile (it does not skip)
    const long long tiles = (long long)a.n * a.nty * a.ntx;
    if (tiles > 0x7fffffffLL) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = pdl_config(L, tiles, LT, s.smem, attr);
    void* args[] = {&a};
    return cudaLaunchKernelExC(&cfg, kernel_of(L), args);
}

}  // namespace sc
