// CUDA-core kernels of the Skip-Conv step:
//   conv_cc    : the convolution of the residual at the open locations only,
//                accumulated into z in place (Eq. 3), as a gathered implicit
//                GEMM on float32 FMAs: M = open output locations (b*b per open
//                block, taken from the compacted list), N = output channels of
//                one group, K = k_h*k_w*(c_in/groups).  Exact to float32
//                rounding for fp32 inputs; serves fp32 layers, strides other
//                than 1, gate blocks other than 8x8 and grouped layers.
//   conv_dw    : the depthwise case (one input channel per output channel),
//                where the contraction is only k_h*k_w long: one thread per
//                channel, residuals read straight from the frames.
//   y_refresh  : y = act(z + shortcut) over the whole frame (layer output handed
//                to the next layer; z itself stays pre-activation, Sec. 3.1).
//   reset_z    : z = bias (state after a reset).
//   pack       : weight repacking at create, and ||w||_1 for the Output-Norm gate.
#include "sc_internal.h"

namespace sc {
namespace {

struct Geom {
    int n, H, W, C, Ho, Wo, Co, KH, KW, stride, pad, b, nby, nbx, cpg, opg;
    int K;                  // k_h * k_w * cpg: contraction length of one output channel
    int n_nt, nt_per_group; // output-channel tiles in all / in one group
};

// Tile of the gathered GEMM: TM open locations x TN output channels, K in
// chunks of TK.  128 threads; thread (tm, tn) owns locations 4*tm..4*tm+3 and
// channels 2*tn, 2*tn+1 of the tile (8 accumulators).  The residual chunk is
// staged as As[location][k] (row stride ASTR, 16-byte aligned rows) and the
// weight chunk as Bs[k][channel]; the next chunk's global loads are issued
// into registers before the current chunk's FMAs.
constexpr int TM = 32, TN = 32, TK = 32, ASTR = TK + 4, CC_THREADS = 128;

template <typename T>
__global__ void __launch_bounds__(CC_THREADS) conv_cc_kernel(const T* __restrict__ xt, const T* __restrict__ xp,
                                                             const float* __restrict__ wcc,
                                                             const int32_t* __restrict__ list,
                                                             const int32_t* __restrict__ counters,
                                                             float* __restrict__ z, T* __restrict__ y, int act, Geom g)
{
    __shared__ __align__(16) float As[TM * ASTR];
    __shared__ __align__(16) float Bs[TK * TN];
    __shared__ int4 loc[TM];   // per tile row: (n*H, top input row, left input col, output pixel or -1)
    const int bb = g.b * g.b;
    const long long n_loc = (long long)counters[0] * bb;
    const long long n_tiles = (n_loc + TM - 1) / TM * g.n_nt;
    const int t = threadIdx.x;
    const int tn = t & 15, tm = t >> 4;     // compute: channels 2tn..2tn+1, locations 4tm..4tm+3
    const int akk = t & 31, am0 = t >> 5;   // residual staging: k = akk, locations am0 + 4j
    const int bnn = t & 31, bk0 = t >> 5;   // weight staging: channel bnn, k = bk0 + 4j
    for (long long tile = blockIdx.x; tile < n_tiles; tile += gridDim.x) {
        const long long mt = tile / g.n_nt;
        const int nt = (int)(tile % g.n_nt);
        const int grp = nt / g.nt_per_group;
        const int o0 = grp * g.opg + (nt % g.nt_per_group) * TN;
        const int o_end = grp * g.opg + g.opg;
        const int c_base = grp * g.cpg;
        __syncthreads();   // the previous tile's epilogue has read loc[]
        if (t < TM) {
            const long long gl = mt * TM + t;
            int4 v = make_int4(0, 0, 0, -1);
            if (gl < n_loc) {
                const int e = (int)(gl / bb), p = (int)(gl - (long long)e * bb);
                const int id = list[e];
                const int bx = id % g.nbx, by = (id / g.nbx) % g.nby, nn = id / (g.nbx * g.nby);
                const int oy = by * g.b + p / g.b, ox = bx * g.b + p % g.b;
                if (oy < g.Ho && ox < g.Wo)
                    v = make_int4(nn * g.H, oy * g.stride - g.pad, ox * g.stride - g.pad,
                                  (nn * g.Ho + oy) * g.Wo + ox);
            }
            loc[t] = v;
        }
        __syncthreads();
        float ra[8], rb[8];
        auto load_chunk = [&](int k0) {
            const int k = k0 + akk;
            const bool kin = k < g.K;
            const int tap = kin ? k / g.cpg : 0;
            const int ci = k - tap * g.cpg;
            const int kh = tap / g.KW, kw = tap - (tap / g.KW) * g.KW;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int4 L = loc[am0 + 4 * j];
                const int iy = L.y + kh, ix = L.z + kw;
                float r = 0.f;
                if (kin && L.w >= 0 && iy >= 0 && iy < g.H && ix >= 0 && ix < g.W) {
                    const size_t off = ((size_t)(L.x + iy) * g.W + ix) * g.C + c_base + ci;
                    r = to_f32(xt[off]) - to_f32(xp[off]);
                }
                ra[j] = r;
            }
            const int o = o0 + bnn;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int kb = k0 + bk0 + 4 * j;
                rb[j] = (kb < g.K && o < o_end) ? __ldg(wcc + (size_t)kb * g.Co + o) : 0.f;
            }
        };
        float acc[4][2];
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[i][0] = acc[i][1] = 0.f;
        load_chunk(0);
        for (int k0 = 0; k0 < g.K; k0 += TK) {
            __syncthreads();   // every thread is done with the previous chunk
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                As[(am0 + 4 * j) * ASTR + akk] = ra[j];
                Bs[(bk0 + 4 * j) * TN + bnn] = rb[j];
            }
            __syncthreads();
            if (k0 + TK < g.K) load_chunk(k0 + TK);
#pragma unroll
            for (int kk = 0; kk < TK; kk += 4) {
                float4 a[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) a[i] = *reinterpret_cast<const float4*>(&As[(tm * 4 + i) * ASTR + kk]);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float2 bv = *reinterpret_cast<const float2*>(&Bs[(kk + q) * TN + tn * 2]);
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const float av = q == 0 ? a[i].x : q == 1 ? a[i].y : q == 2 ? a[i].z : a[i].w;
                        acc[i][0] = fmaf(av, bv.x, acc[i][0]);
                        acc[i][1] = fmaf(av, bv.y, acc[i][1]);
                    }
                }
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int4 L = loc[tm * 4 + i];
            if (L.w < 0) continue;
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                const int o = o0 + tn * 2 + j;
                if (o >= o_end) continue;
                const size_t zo = (size_t)L.w * g.Co + o;
                const float zv = z[zo] + acc[i][j];
                z[zo] = zv;
                if (y) y[zo] = from_f32<T>(activate(zv, act));
            }
        }
    }
}

// Depthwise layers: one work unit = one output row of an open block; the
// block's threads stride over the channels and walk the row's locations.
template <typename T>
__global__ void __launch_bounds__(256) conv_dw_kernel(const T* __restrict__ xt, const T* __restrict__ xp,
                                                      const float* __restrict__ wcc,
                                                      const int32_t* __restrict__ list,
                                                      const int32_t* __restrict__ counters, float* __restrict__ z,
                                                      T* __restrict__ y, int act, Geom g)
{
    const long long units = (long long)counters[0] * g.b;
    for (long long u = blockIdx.x; u < units; u += gridDim.x) {
        const int e = (int)(u / g.b), row = (int)(u - (long long)e * g.b);
        const int id = list[e];
        const int bx = id % g.nbx, by = (id / g.nbx) % g.nby, nn = id / (g.nbx * g.nby);
        const int oy = by * g.b + row;
        if (oy >= g.Ho) continue;
        const int iy0 = oy * g.stride - g.pad;
        const int bw = min(g.b, g.Wo - bx * g.b);
        for (int c = threadIdx.x; c < g.C; c += blockDim.x) {
            for (int j = 0; j < bw; ++j) {
                const int ox = bx * g.b + j;
                const int ix0 = ox * g.stride - g.pad;
                float acc = 0.f;
                for (int kh = 0; kh < g.KH; ++kh) {
                    const int iy = iy0 + kh;
                    if (iy < 0 || iy >= g.H) continue;
                    for (int kw = 0; kw < g.KW; ++kw) {
                        const int ix = ix0 + kw;
                        if (ix < 0 || ix >= g.W) continue;
                        const size_t off = (((size_t)nn * g.H + iy) * g.W + ix) * g.C + c;
                        acc = fmaf(__ldg(wcc + (size_t)(kh * g.KW + kw) * g.Co + c), to_f32(xt[off]) - to_f32(xp[off]),
                                   acc);
                    }
                }
                const size_t zo = (((size_t)nn * g.Ho + oy) * g.Wo + ox) * g.Co + c;
                const float zv = z[zo] + acc;
                z[zo] = zv;
                if (y) y[zo] = from_f32<T>(activate(zv, act));
            }
        }
    }
}

template <typename T>
__global__ void y_refresh_kernel(const float* __restrict__ z, const T* __restrict__ sc, T* __restrict__ y,
                                 long long count, int act)
{
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < count;
         i += (long long)gridDim.x * blockDim.x) {
        const float v = z[i] + (sc ? to_f32(sc[i]) : 0.f);
        y[i] = from_f32<T>(activate(v, act));
    }
}

__global__ void reset_z_kernel(float* __restrict__ z, const float* __restrict__ bias, long long count, int co)
{
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < count;
         i += (long long)gridDim.x * blockDim.x)
        z[i] = bias ? bias[i % co] : 0.f;
}

// OIHW (dtype) -> w_cc [KH][KW][cpg][Co] fp32 (row k = (kh*KW + kw)*cpg + ci of the
// CUDA-core GEMM's weight operand) and, when w_tc != NULL,
// w_tc [co_pad][KH*KW*ci_pad] bf16 (K index = (kh*KW + kw)*ci_pad + ci).
template <typename T>
__global__ void pack_weights_kernel(const T* __restrict__ w, float* __restrict__ wcc, __nv_bfloat16* __restrict__ wtc,
                                    double* __restrict__ l1, int Co, int cpg, int KH, int KW, int ci_pad)
{
    const long long total = (long long)Co * cpg * KH * KW;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int kw = (int)(i % KW);
        const int kh = (int)((i / KW) % KH);
        const int ci = (int)((i / (KW * KH)) % cpg);
        const int o = (int)(i / ((long long)KW * KH * cpg));
        const float v = to_f32(w[i]);
        wcc[((size_t)(kh * KW + kw) * cpg + ci) * Co + o] = v;
        if (wtc) wtc[(size_t)o * KH * KW * ci_pad + (size_t)(kh * KW + kw) * ci_pad + ci] = __float2bfloat16_rn(v);
        atomicAdd(l1, (double)fabsf(v));
    }
}

}  // namespace

cudaError_t launch_conv_cc(const Layer& L, const void* x_t, const void* x_prev)
{
    Geom g;
    g.n = L.p.n_streams; g.H = L.p.h; g.W = L.p.w; g.C = L.p.c_in; g.Ho = L.ho; g.Wo = L.wo; g.Co = L.p.c_out;
    g.KH = L.p.k_h; g.KW = L.p.k_w; g.stride = L.p.stride; g.pad = L.p.pad; g.b = L.p.block;
    g.nby = L.nby; g.nbx = L.nbx; g.cpg = L.cpg; g.opg = L.opg;
    g.K = L.p.k_h * L.p.k_w * L.cpg;
    g.nt_per_group = (L.opg + TN - 1) / TN;
    g.n_nt = g.nt_per_group * L.p.groups;
    const long long nblocks = (long long)L.p.n_streams * L.nby * L.nbx;
    const bool depthwise = L.cpg == 1 && L.opg == 1;
    // y is written here only when there is no shortcut (otherwise y_refresh rewrites the frame)
    if (depthwise) {
        const long long units = nblocks * L.p.block;
        const long long cap = (long long)L.num_sms * 4;
        const int grid = (int)(units < cap ? units : cap);
        if (L.p.dtype == SKIPCONV_BF16)
            conv_dw_kernel<__nv_bfloat16><<<grid, 256, 0, L.stream>>>(
                (const __nv_bfloat16*)x_t, (const __nv_bfloat16*)x_prev, L.w_cc, L.list, step_count(L), L.z,
                (__nv_bfloat16*)L.y, L.p.activation, g);
        else
            conv_dw_kernel<float><<<grid, 256, 0, L.stream>>>((const float*)x_t, (const float*)x_prev, L.w_cc, L.list,
                                                              step_count(L), L.z, (float*)L.y, L.p.activation, g);
        return cudaGetLastError();
    }
    const long long bb = (long long)L.p.block * L.p.block;
    const long long tiles = (nblocks * bb + TM - 1) / TM * g.n_nt;
    const long long cap = (long long)L.num_sms * 2;
    const int grid = (int)(tiles < cap ? tiles : cap);
    if (L.p.dtype == SKIPCONV_BF16)
        conv_cc_kernel<__nv_bfloat16><<<grid, CC_THREADS, 0, L.stream>>>(
            (const __nv_bfloat16*)x_t, (const __nv_bfloat16*)x_prev, L.w_cc, L.list, step_count(L), L.z,
            (__nv_bfloat16*)L.y, L.p.activation, g);
    else
        conv_cc_kernel<float><<<grid, CC_THREADS, 0, L.stream>>>((const float*)x_t, (const float*)x_prev, L.w_cc,
                                                                 L.list, step_count(L), L.z, (float*)L.y,
                                                                 L.p.activation, g);
    return cudaGetLastError();
}

cudaError_t launch_y_refresh(const Layer& L, const void* shortcut)
{
    const long long count = (long long)L.p.n_streams * L.ho * L.wo * L.p.c_out;
    long long blocks = (count + 255) / 256;
    const long long cap = (long long)L.num_sms * 8;
    const int grid = (int)(blocks < cap ? blocks : cap);
    if (L.p.dtype == SKIPCONV_BF16)
        y_refresh_kernel<__nv_bfloat16><<<grid, 256, 0, L.stream>>>(L.z, (const __nv_bfloat16*)shortcut,
                                                                   (__nv_bfloat16*)L.y, count, L.p.activation);
    else
        y_refresh_kernel<float><<<grid, 256, 0, L.stream>>>(L.z, (const float*)shortcut, (float*)L.y, count,
                                                           L.p.activation);
    return cudaGetLastError();
}

cudaError_t launch_reset_z(const Layer& L)
{
    const long long count = (long long)L.p.n_streams * L.ho * L.wo * L.p.c_out;
    long long blocks = (count + 255) / 256;
    const long long cap = (long long)L.num_sms * 8;
    const int grid = (int)(blocks < cap ? blocks : cap);
    reset_z_kernel<<<grid, 256, 0, L.stream>>>(L.z, L.bias, count, L.p.c_out);
    return cudaGetLastError();
}

// Open blocks of z into a packed buffer: CTA j takes blocks j, j + grid, ... of the step's list;
// each copies the block's b x b x c_out values (16-byte vectors when c_out is a multiple of 4),
// zeros past the frame's edge.  CTA 0 also copies the count and the list.
__global__ void gather_open_blocks_kernel(const float* __restrict__ z, const int32_t* __restrict__ list,
                                          const int32_t* __restrict__ count, float* __restrict__ zb,
                                          int32_t* __restrict__ list_out, int32_t* __restrict__ count_out, int Ho,
                                          int Wo, int Co, int b, int nby, int nbx)
{
    const int cnt = *count;
    if (blockIdx.x == 0) {
        for (int i = threadIdx.x; i < cnt; i += blockDim.x) list_out[i] = list[i];
        if (threadIdx.x == 0) *count_out = cnt;
    }
    const int row = b * Co;   // floats of one block row
    for (int i = blockIdx.x; i < cnt; i += gridDim.x) {
        const int id = list[i];
        const int bx = id % nbx, by = (id / nbx) % nby, n = id / (nbx * nby);
        float* dst = zb + (size_t)i * b * row;
        if ((Co & 3) == 0) {
            const int q4 = row / 4;
            for (int e = threadIdx.x; e < b * q4; e += blockDim.x) {
                const int r = e / q4, q = e - r * q4;
                const int oy = by * b + r, ox = bx * b + (4 * q) / Co;
                float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                if (oy < Ho && ox < Wo)
                    v = *reinterpret_cast<const float4*>(z + (((size_t)n * Ho + oy) * Wo + ox) * Co + (4 * q) % Co);
                reinterpret_cast<float4*>(dst + (size_t)r * row)[q] = v;
            }
        } else {
            for (int e = threadIdx.x; e < b * row; e += blockDim.x) {
                const int r = e / row, q = e - r * row;
                const int oy = by * b + r, ox = bx * b + q / Co;
                dst[e] = (oy < Ho && ox < Wo) ? z[(((size_t)n * Ho + oy) * Wo + ox) * Co + q % Co] : 0.f;
            }
        }
    }
}

cudaError_t launch_gather_open_blocks(const Layer& L, const int32_t* count, float* zb, int32_t* list_out,
                                      int32_t* count_out)
{
    const int grid = L.num_sms * 4;
    gather_open_blocks_kernel<<<grid, 256, 0, L.stream>>>(L.z, L.list, count, zb, list_out, count_out, L.ho,
                                                         L.wo, L.p.c_out, L.p.block, L.nby, L.nbx);
    return cudaGetLastError();
}

cudaError_t launch_pack_weights(Layer& L, const void* w_oihw, double* w_l1_dev)
{
    const long long total = (long long)L.p.c_out * L.cpg * L.p.k_h * L.p.k_w;
    long long blocks = (total + 255) / 256;
    const int grid = (int)(blocks < 4096 ? blocks : 4096);
    if (L.p.dtype == SKIPCONV_BF16)
        pack_weights_kernel<__nv_bfloat16><<<grid, 256, 0, L.stream>>>((const __nv_bfloat16*)w_oihw, L.w_cc, L.w_tc,
                                                                      w_l1_dev, L.p.c_out, L.cpg, L.p.k_h,
                                                                      L.p.k_w, L.ci_pad);
    else
        pack_weights_kernel<float><<<grid, 256, 0, L.stream>>>((const float*)w_oihw, L.w_cc, L.w_tc, w_l1_dev,
                                                              L.p.c_out, L.cpg, L.p.k_h, L.p.k_w, L.ci_pad);
    return cudaGetLastError();
}

}  // namespace sc
