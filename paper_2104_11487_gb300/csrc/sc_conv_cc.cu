// CUDA-core kernels of the Skip-Conv step:
//   conv_cc    : direct convolution of the residual over the open blocks only,
//                accumulated into z in place (Eq. 3); float32 FMA, so it is exact
//                to float32 rounding for fp32 inputs and serves grouped /
//                depthwise layers, where the contraction is too short for MMAs.
//   y_refresh  : y = act(z + shortcut) over the whole frame (layer output handed
//                to the next layer; z itself stays pre-activation, Sec. 3.1).
//   reset_z    : z = bias (state after a reset).
//   pack       : weight repacking at create, and ||w||_1 for the Output-Norm gate.
#include "sc_internal.h"

namespace sc {
namespace {

struct Geom {
    int n, H, W, C, Ho, Wo, Co, KH, KW, stride, pad, b, nby, nbx, cpg, opg, HH, WW;
};

template <typename T>
__global__ void __launch_bounds__(256) conv_cc_kernel(const T* __restrict__ xt, const T* __restrict__ xp,
                                                      const float* __restrict__ wcc,
                                                      const int32_t* __restrict__ list,
                                                      const int32_t* __restrict__ counters, float* __restrict__ z,
                                                      T* __restrict__ y, int act, Geom g)
{
    extern __shared__ float rs[];  // residual halo tile [HH][WW][C], float32
    const int count = counters[0];
    const int tile = g.HH * g.WW * g.C;
    for (int e = blockIdx.x; e < count; e += gridDim.x) {
        const int id = list[e];
        const int bx = id % g.nbx;
        const int by = (id / g.nbx) % g.nby;
        const int n = id / (g.nbx * g.nby);
        const int y0 = by * g.b * g.stride - g.pad;
        const int x0 = bx * g.b * g.stride - g.pad;
        __syncthreads();
        for (int idx = threadIdx.x; idx < tile; idx += blockDim.x) {
            const int c = idx % g.C;
            const int t2 = idx / g.C;
            const int ww = t2 % g.WW;
            const int hh = t2 / g.WW;
            const int yy = y0 + hh, xx = x0 + ww;
            float r = 0.f;
            if (yy >= 0 && yy < g.H && xx >= 0 && xx < g.W) {
                const size_t off = (((size_t)n * g.H + yy) * g.W + xx) * g.C + c;
                r = to_f32(xt[off]) - to_f32(xp[off]);
            }
            rs[idx] = r;
        }
        __syncthreads();
        const int bh = min(g.b, g.Ho - by * g.b), bw = min(g.b, g.Wo - bx * g.b);
        const int pairs = g.b * g.b * g.Co;
        for (int idx = threadIdx.x; idx < pairs; idx += blockDim.x) {
            const int o = idx % g.Co;
            const int pp = idx / g.Co;
            const int i = pp / g.b, j = pp % g.b;
            if (i >= bh || j >= bw) continue;
            const int c0 = (o / g.opg) * g.cpg;
            float acc = 0.f;
            for (int ci = 0; ci < g.cpg; ++ci)
                for (int kh = 0; kh < g.KH; ++kh)
                    for (int kw = 0; kw < g.KW; ++kw)
                        acc = fmaf(__ldg(wcc + ((size_t)(ci * g.KH + kh) * g.KW + kw) * g.Co + o),
                                   rs[((i * g.stride + kh) * g.WW + (j * g.stride + kw)) * g.C + c0 + ci], acc);
            const size_t zo = (((size_t)n * g.Ho + by * g.b + i) * g.Wo + bx * g.b + j) * g.Co + o;
            const float zv = z[zo] + acc;
            z[zo] = zv;
            if (y) y[zo] = from_f32<T>(activate(zv, act));
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

// OIHW (dtype) -> w_cc [cpg][KH][KW][Co] fp32 and, when w_tc != NULL,
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
        wcc[((size_t)(ci * KH + kh) * KW + kw) * Co + o] = v;
        if (wtc) wtc[(size_t)o * KH * KW * ci_pad + (size_t)(kh * KW + kw) * ci_pad + ci] = __float2bfloat16_rn(v);
        atomicAdd(l1, (double)fabsf(v));
    }
}

}  // namespace

size_t conv_cc_smem_bytes(const Layer& L)
{
    const int HH = (L.p.block - 1) * L.p.stride + L.p.k_h;
    const int WW = (L.p.block - 1) * L.p.stride + L.p.k_w;
    return (size_t)HH * WW * L.p.c_in * sizeof(float);
}

cudaError_t launch_conv_cc(const Layer& L, const void* x_t, const void* x_prev)
{
    Geom g;
    g.n = L.p.n_streams; g.H = L.p.h; g.W = L.p.w; g.C = L.p.c_in; g.Ho = L.ho; g.Wo = L.wo; g.Co = L.p.c_out;
    g.KH = L.p.k_h; g.KW = L.p.k_w; g.stride = L.p.stride; g.pad = L.p.pad; g.b = L.p.block;
    g.nby = L.nby; g.nbx = L.nbx; g.cpg = L.cpg; g.opg = L.opg;
    g.HH = (L.p.block - 1) * L.p.stride + L.p.k_h;
    g.WW = (L.p.block - 1) * L.p.stride + L.p.k_w;
    const size_t smem = conv_cc_smem_bytes(L);
    const long long nblocks = (long long)L.p.n_streams * L.nby * L.nbx;
    const int per_sm = smem > 100 * 1024 ? 1 : (smem > 48 * 1024 ? 2 : 4);
    const long long cap = (long long)L.num_sms * per_sm;
    const int grid = (int)(nblocks < cap ? nblocks : cap);
    // y is written here only when there is no shortcut (otherwise y_refresh rewrites the frame)
    if (L.p.dtype == SKIPCONV_BF16) {
        auto k = conv_cc_kernel<__nv_bfloat16>;
        cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        k<<<grid, 256, smem, L.stream>>>((const __nv_bfloat16*)x_t, (const __nv_bfloat16*)x_prev, L.w_cc, L.list,
                                         step_count(L), L.z, (__nv_bfloat16*)L.y, L.p.activation, g);
    } else {
        auto k = conv_cc_kernel<float>;
        cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        k<<<grid, 256, smem, L.stream>>>((const float*)x_t, (const float*)x_prev, L.w_cc, L.list, step_count(L), L.z,
                                         (float*)L.y, L.p.activation, g);
    }
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
