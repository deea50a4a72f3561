// Tensor-core convolution of the open blocks (Eq. 3's w * r_t on the gated
// locations), as a gathered implicit GEMM on sm_103a tcgen05.
//
// One work unit = (open 8x8 block, tile of 128 output channels):
//     D[co][p] = sum_k W[co][k] * R[p][k],   M = 128 (co), N = 64 (p), K = k_h*k_w*ci_pad
// with k = (tap, input channel).  The residual operand is never expanded to
// im2col: TMA loads the (8+k_h-1) x (8+k_w-1) halo of x_t and of x_{t-1}
// straight into the no-swizzle K-major canonical layout
//     [8-channel group][halo row][halo col][8 channels]   (16-byte core-matrix rows)
// (zero fill outside the frame = the convolution's zero padding), four
// residual warps overwrite the x_t copy with bf16(x_t - x_{t-1}), and the
// operand of tap (kh, kw) is the same buffer seen through a descriptor whose
// start is shifted by (kh*WW + kw)*16 bytes: the 8 pixels of an output row
// are 8 consecutive 16-byte rows (a core matrix), output rows are WW*16
// bytes apart (stride-dimension offset) and 8-channel groups HH*WW*16 bytes
// apart (leading-dimension offset).  Weights come in 128 x 64 tiles through
// TMA with the 128-byte swizzle.  The fp32 accumulator lives in TMEM
// (2 x 64 columns, double-buffered across units); four epilogue warps read it
// with tcgen05.ld and add it into z in place (the scatter-accumulate of
// Eq. 3), optionally writing y = act(z).
//
// Warp roles: 0-3 epilogue, 4-7 residual, 8 weight-tile producer, 9 MMA issuer,
// 10 halo-tile producer (separate so that the weight stream never waits on
// the halo ring, and vice versa).
#include <math.h>
#include <stdlib.h>

#include "sc_internal.h"
#include "sc_ptx.cuh"
#include "sc_tc_common.cuh"

namespace sc {
namespace {

constexpr int TC_ASTAGES = 8;
constexpr int TC_XSTAGES = 2;
constexpr int TC_THREADS = 352;
constexpr int TC_ABYTES = TC_M * TC_CK * 2;  // 16 KiB weight tile
constexpr uint32_t TC_TMEM_COLS = 2 * TC_N;
constexpr uint64_t WAIT_LIMIT_NS = 1000000000ull;

struct TcArgs {
    const int32_t* list;
    const int32_t* counters;
    float* z;
    __nv_bfloat16* y;
    int* err;
    int act;
    int H, W, Ho, Wo, Co, KH, KW, pad, nby, nbx;
    int n_ct, n_chunks, HH, WW, taps, ci_pad;
    int x5d;
    int z_tma;   // 1: z += D through a TMA reduce-add (no y); 0: load, add, store (and y)
};

struct Bars {
    uint64_t x_full[TC_XSTAGES], r_ready[TC_XSTAGES], x_empty[TC_XSTAGES];
    uint64_t a_full[TC_ASTAGES], a_empty[TC_ASTAGES];
    uint64_t acc_full[2], acc_empty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};

size_t tc_smem_bytes(int HH, int WW)
{
    return 1024 + (size_t)TC_ASTAGES * TC_ABYTES + (size_t)TC_XSTAGES * 2 * x_tile_bytes(HH, WW) + TC_ZBYTES +
           sizeof(Bars);
}

__device__ __forceinline__ void decode_unit(const TcArgs& a, int u, int& n, int& by, int& bx, int& ct)
{
    const int e = u / a.n_ct;
    ct = u - e * a.n_ct;
    const int id = a.list[e];
    bx = id % a.nbx;
    by = (id / a.nbx) % a.nby;
    n = id / (a.nbx * a.nby);
}

__global__ void __launch_bounds__(TC_THREADS, 1)
conv_tc_kernel(const __grid_constant__ CUtensorMap tm_xt, const __grid_constant__ CUtensorMap tm_xp,
               const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_z, const TcArgs a)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = ptx::align_smem_1024(smem_raw);
    const int XB = x_tile_bytes(a.HH, a.WW);
    uint8_t* sA = smem;
    uint8_t* sX = smem + TC_ASTAGES * TC_ABYTES;
    float* sZ = (float*)(sX + TC_XSTAGES * 2 * XB);
    Bars* bars = (Bars*)((uint8_t*)sZ + TC_ZBYTES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int units = a.counters[0] * a.n_ct;
    if ((int)blockIdx.x >= units) return;

    if (threadIdx.x == 0) {
        for (int s = 0; s < TC_XSTAGES; ++s) {
            ptx::mbar_init(ptx::smem_u32(&bars->x_full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&bars->r_ready[s]), 4);
            ptx::mbar_init(ptx::smem_u32(&bars->x_empty[s]), 1);
        }
        for (int s = 0; s < TC_ASTAGES; ++s) {
            ptx::mbar_init(ptx::smem_u32(&bars->a_full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&bars->a_empty[s]), 1);
        }
        for (int s = 0; s < 2; ++s) {
            ptx::mbar_init(ptx::smem_u32(&bars->acc_full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&bars->acc_empty[s]), 4);
        }
        ptx::mbar_init(ptx::smem_u32(&bars->drain), 1);
        bars->abort = 0;
        ptx::fence_mbar_init();
    }
    if (warp == 9) {
        ptx::tmem_alloc(ptx::smem_u32(&bars->tmem_base), TC_TMEM_COLS);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort = &bars->abort;

    if (warp == 8 || warp == 10) {
        // ------------------------------------------------ TMA producers
        if (lane == 0) {
            const bool halo = warp == 10;
            ptx::prefetch_tmap(halo ? &tm_xt : &tm_w);
            if (halo) ptx::prefetch_tmap(&tm_xp);
            int st = 0;
            uint32_t ph = 0;
            uint32_t issue_ph[TC_ASTAGES] = {};
            uint32_t issued = 0;  // bit per stage: a load was issued there
            bool ok = true;
            for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
                int n, by, bx, ct;
                decode_unit(a, u, n, by, bx, ct);
                const int y0 = by * 8 - a.pad, x0 = bx * 8 - a.pad;
                for (int c = 0; c < a.n_chunks && ok; ++c) {
                    if (halo) {
                        const uint32_t xf = ptx::smem_u32(&bars->x_full[st]);
                        if (!(ok = ptx::mbar_wait(ptx::smem_u32(&bars->x_empty[st]), ph ^ 1, abort, a.err,
                                                  WAIT_LIMIT_NS)))
                            break;
                        ptx::mbar_arrive_expect_tx(xf, 2 * XB);
                        const uint32_t dst = ptx::smem_u32(sX + st * 2 * XB);
                        if (a.x5d) {
                            ptx::tma_load_5d(dst, &tm_xt, xf, 0, x0, y0, c * 8, n);
                            ptx::tma_load_5d(dst + XB, &tm_xp, xf, 0, x0, y0, c * 8, n);
                        } else {
                            const int gb = a.HH * a.WW * 16;
                            for (int g = 0; g < 8; ++g) {
                                ptx::tma_load_4d(dst + g * gb, &tm_xt, xf, (c * 8 + g) * 8, x0, y0, n);
                                ptx::tma_load_4d(dst + XB + g * gb, &tm_xp, xf, (c * 8 + g) * 8, x0, y0, n);
                            }
                        }
                        issue_ph[st] = ph;
                        issued |= 1u << st;
                        if (++st == TC_XSTAGES) { st = 0; ph ^= 1; }
                    } else {
                        for (int t = 0; t < a.taps; ++t) {
                            const uint32_t af = ptx::smem_u32(&bars->a_full[st]);
                            if (!(ok = ptx::mbar_wait(ptx::smem_u32(&bars->a_empty[st]), ph ^ 1, abort, a.err,
                                                      WAIT_LIMIT_NS)))
                                break;
                            ptx::mbar_arrive_expect_tx(af, TC_ABYTES);
                            ptx::tma_load_2d(ptx::smem_u32(sA + st * TC_ABYTES), &tm_w, af,
                                             t * a.ci_pad + c * TC_CK, ct * TC_M);
                            issue_ph[st] = ph;
                            issued |= 1u << st;
                            if (++st == TC_ASTAGES) { st = 0; ph ^= 1; }
                        }
                    }
                }
            }
            if (!ok) {
                // let every copy this thread started land before the CTA exits
                const int nst = halo ? TC_XSTAGES : TC_ASTAGES;
                for (int s2 = 0; s2 < nst; ++s2)
                    if (issued & (1u << s2))
                        ptx::mbar_wait(ptx::smem_u32(halo ? &bars->x_full[s2] : &bars->a_full[s2]), issue_ph[s2],
                                       nullptr, nullptr, WAIT_LIMIT_NS);
            }
        }
    } else if (warp == 9) {
        // ---------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = ptx::idesc_bf16_f32(TC_M, TC_N);
            const uint32_t sbo = a.WW * 16, lbo = a.HH * a.WW * 16;
            int xs = 0, as = 0, acc = 0;
            uint32_t xph = 0, aph = 0, accph = 0;
            bool ok = true, issued = false;
            for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
                if (!(ok = ptx::mbar_wait(ptx::smem_u32(&bars->acc_empty[acc]), accph ^ 1, abort, a.err,
                                          WAIT_LIMIT_NS)))
                    break;
                ptx::tc_fence_after();
                const uint32_t d = tmem + acc * TC_N;
                for (int c = 0; c < a.n_chunks && ok; ++c) {
                    if (!(ok = ptx::mbar_wait(ptx::smem_u32(&bars->r_ready[xs]), xph, abort, a.err, WAIT_LIMIT_NS)))
                        break;
                    ptx::tc_fence_after();
                    const uint32_t xbase = ptx::smem_u32(sX + xs * 2 * XB);
                    for (int t = 0; t < a.taps; ++t) {
                        const int kh = t / a.KW, kw = t - (t / a.KW) * a.KW;
                        if (!(ok = ptx::mbar_wait(ptx::smem_u32(&bars->a_full[as]), aph, abort, a.err,
                                                  WAIT_LIMIT_NS)))
                            break;
                        ptx::tc_fence_after();
                        const uint32_t abase = ptx::smem_u32(sA + as * TC_ABYTES);
#pragma unroll
                        for (int q = 0; q < TC_CK / 16; ++q) {
                            const uint64_t ad = ptx::smem_desc(abase + q * 32, 16, 1024, 2);
                            const uint64_t bd =
                                ptx::smem_desc(xbase + ((2 * q * a.HH + kh) * a.WW + kw) * 16, lbo, sbo, 0);
                            ptx::mma_bf16(d, ad, bd, idesc, (c | t | q) != 0);
                        }
                        issued = true;
                        ptx::mma_commit(ptx::smem_u32(&bars->a_empty[as]));
                        if (++as == TC_ASTAGES) { as = 0; aph ^= 1; }
                    }
                    if (!ok) break;
                    ptx::mma_commit(ptx::smem_u32(&bars->x_empty[xs]));
                    if (++xs == TC_XSTAGES) { xs = 0; xph ^= 1; }
                }
                if (!ok) break;
                ptx::mma_commit(ptx::smem_u32(&bars->acc_full[acc]));
                if (++acc == 2) { acc = 0; accph ^= 1; }
            }
            if (!ok && issued) {
                // every MMA issued so far must finish before TMEM is released
                ptx::mma_commit(ptx::smem_u32(&bars->drain));
                ptx::mbar_wait(ptx::smem_u32(&bars->drain), 0, nullptr, nullptr, WAIT_LIMIT_NS);
            }
        }
    } else if (warp >= 4) {
        // ------------------------------------- residual r = x_t - x_{t-1}
        const int tid = threadIdx.x - 128;
        int xs = 0;
        uint32_t xph = 0;
        bool ok = true;
        for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
            for (int c = 0; c < a.n_chunks; ++c) {
                if (!(ok = ptx::mbar_wait(ptx::smem_u32(&bars->x_full[xs]), xph, abort, a.err, WAIT_LIMIT_NS)))
                    break;
                uint4* xt = (uint4*)(sX + xs * 2 * XB);
                const uint4* xp = (const uint4*)(sX + xs * 2 * XB + XB);
                const int nv = XB / 16;
                for (int v = tid; v < nv; v += 128) xt[v] = bf16x8_sub(xt[v], xp[v]);
                ptx::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&bars->r_ready[xs]));
                if (++xs == TC_XSTAGES) { xs = 0; xph ^= 1; }
            }
        }
    } else {
        // ------------------------------------------- epilogue: z += D
        const int tid = threadIdx.x;  // 0..127
        int acc = 0;
        uint32_t accph = 0;
        for (int u = blockIdx.x; u < units; u += gridDim.x) {
            int n, by, bx, ct;
            decode_unit(a, u, n, by, bx, ct);
            if (!ptx::mbar_wait(ptx::smem_u32(&bars->acc_full[acc]), accph, abort, a.err, WAIT_LIMIT_NS)) break;
            ptx::tc_fence_after();
            uint32_t r0[32], r1[32];
            const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + acc * TC_N;
            ptx::tmem_ld_32x32b_x32(taddr, r0);
            ptx::tmem_ld_32x32b_x32(taddr + 32, r1);
            ptx::tmem_wait_ld();
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&bars->acc_empty[acc]));
            if (++acc == 2) { acc = 0; accph ^= 1; }
            const int col = warp * 32 + lane;  // output channel within the tile
            if (a.z_tma) {
                // stage D as [pixel][channel] fp32 and add it into z at L2
                if (tid == 0) ptx::bulk_wait_group_read0();
                ptx::named_bar_sync(1, 128);
#pragma unroll
                for (int p = 0; p < 32; ++p) {
                    sZ[p * TC_M + col] = __uint_as_float(r0[p]);
                    sZ[(p + 32) * TC_M + col] = __uint_as_float(r1[p]);
                }
                ptx::fence_proxy_async_smem();
                ptx::named_bar_sync(1, 128);
                if (tid == 0) {
                    ptx::tma_reduce_add_4d(&tm_z, ptx::smem_u32(sZ), ct * TC_M, bx * 8, by * 8, n);
                    ptx::bulk_commit_group();
                }
            } else {
                const int co = ct * TC_M + col;
                if (co < a.Co) {
                    float* zb = a.z + ((size_t)n * a.Ho * a.Wo) * a.Co + co;
                    __nv_bfloat16* yb = a.y ? a.y + ((size_t)n * a.Ho * a.Wo) * a.Co + co : nullptr;
                    // one output row (8 pixels) at a time: 8 loads in flight, then 8 stores
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const int oy = by * 8 + i;
                        if (oy >= a.Ho) break;
                        float* zr = zb + ((size_t)oy * a.Wo + bx * 8) * a.Co;
                        float zv[8];
#pragma unroll
                        for (int j = 0; j < 8; ++j) zv[j] = (bx * 8 + j < a.Wo) ? zr[(size_t)j * a.Co] : 0.f;
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            if (bx * 8 + j < a.Wo) {
                                const int q = i * 8 + j;
                                const float v = zv[j] + __uint_as_float(q < 32 ? r0[q & 31] : r1[q & 31]);
                                zr[(size_t)j * a.Co] = v;
                                if (yb) yb[((size_t)oy * a.Wo + bx * 8 + j) * a.Co] = __float2bfloat16_rn(activate(v, a.act));
                            }
                        }
                    }
                }
            }
        }
        if (a.z_tma && tid == 0) ptx::bulk_wait_group0();
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        __syncwarp();
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, TC_TMEM_COLS);
    }
}

// ------------------------------------------------------------ tensor maps
}  // namespace

bool tc_encode_x_map(CUtensorMap* m, const void* base, const Layer& L, bool five_d)
{
    EncodeTiledFn enc = encode_tiled_fn();
    if (!enc) return false;
    const int HH = 8 + L.p.k_h - 1, WW = 8 + L.p.k_w - 1;
    const cuuint64_t C = L.p.c_in, W = L.p.w, H = L.p.h, N = L.p.n_streams;
    cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    CUresult r;
    if (five_d) {
        // dims (inner -> outer): 8 channels, w, h, channel group, stream
        cuuint64_t dims[5] = {8, W, H, C / 8, N};
        cuuint64_t strides[4] = {C * 2, W * C * 2, 16, H * W * C * 2};
        cuuint32_t box[5] = {8, (cuuint32_t)WW, (cuuint32_t)HH, 8, 1};
        r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    } else {
        cuuint64_t dims[4] = {C, W, H, N};
        cuuint64_t strides[3] = {C * 2, W * C * 2, H * W * C * 2};
        cuuint32_t box[4] = {8, (cuuint32_t)WW, (cuuint32_t)HH, 1};
        r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    }
    return r == CUDA_SUCCESS;
}

bool tc_encode_z_map(CUtensorMap* m, const Layer& L)
{
    EncodeTiledFn enc = encode_tiled_fn();
    if (!enc || L.p.c_out % 4) return false;
    const cuuint64_t Co = L.p.c_out, Wo = L.wo, Ho = L.ho, N = L.p.n_streams;
    cuuint64_t dims[4] = {Co, Wo, Ho, N};
    cuuint64_t strides[3] = {Co * 4, Wo * Co * 4, Ho * Wo * Co * 4};
    cuuint32_t box[4] = {TC_M, 8, 8, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, L.z, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool conv_tc_supported(const skipconv_params& p, const char** why)
{
    if (p.dtype != SKIPCONV_BF16) return *why = "needs bf16 data", false;
    if (p.groups != 1) return *why = "grouped convolution", false;
    if (p.stride != 1) return *why = "stride other than 1", false;
    if (p.block != 8) return *why = "gate block other than 8x8", false;
    if (p.c_in % 8) return *why = "c_in not a multiple of 8", false;
    if (p.k_h > 7 || p.k_w > 7) return *why = "kernel larger than 7", false;
    if (tc_smem_bytes(8 + p.k_h - 1, 8 + p.k_w - 1) > 227 * 1024) return *why = "shared memory", false;
    return true;
}

cudaError_t conv_tc_prepare(Layer& L)
{
    EncodeTiledFn enc = encode_tiled_fn();
    if (!enc) {
        set_error("cuTensorMapEncodeTiled unavailable");
        return cudaErrorNotSupported;
    }
    L.tc_x5d = 1;
    if (!tc_encode_x_map(&L.tmap_xbuf[0], L.xbuf[0], L, true) || !tc_encode_x_map(&L.tmap_xbuf[1], L.xbuf[1], L, true)) {
        L.tc_x5d = 0;
        if (!tc_encode_x_map(&L.tmap_xbuf[0], L.xbuf[0], L, false) || !tc_encode_x_map(&L.tmap_xbuf[1], L.xbuf[1], L, false)) {
            set_error("tensor map of the state frames rejected");
            return cudaErrorInvalidValue;
        }
    }
    const cuuint64_t KT = (cuuint64_t)L.p.k_h * L.p.k_w * L.ci_pad;
    cuuint64_t dims[2] = {KT, (cuuint64_t)L.co_pad};
    cuuint64_t strides[1] = {KT * 2};
    cuuint32_t box[2] = {TC_CK, TC_M};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(&L.tmap_w, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, L.w_tc, dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        set_error("tensor map of the weights rejected (%d)", (int)r);
        return cudaErrorInvalidValue;
    }
    L.tc_z_tma = tc_encode_z_map(&L.tmap_z, L) ? 1 : 0;
    const int HH = 8 + L.p.k_h - 1, WW = 8 + L.p.k_w - 1;
    return ensure_dynamic_smem((const void*)conv_tc_kernel, tc_smem_bytes(HH, WW));
}

cudaError_t launch_conv_tc(const Layer& L, const void* x_t, const void* x_prev, int prev_index)
{
    (void)x_prev;
    alignas(64) CUtensorMap tm_xt;
    if (!tc_encode_x_map(&tm_xt, x_t, L, L.tc_x5d != 0)) {
        set_error("tensor map of x_t rejected");
        return cudaErrorInvalidValue;
    }
    TcArgs a;
    a.list = L.list;
    a.counters = step_count(L);
    a.z = L.z;
    a.y = (__nv_bfloat16*)L.y;
    a.err = L.err_dev;
    a.act = L.p.activation;
    a.H = L.p.h;
    a.W = L.p.w;
    a.Ho = L.ho;
    a.Wo = L.wo;
    a.Co = L.p.c_out;
    a.KH = L.p.k_h;
    a.KW = L.p.k_w;
    a.pad = L.p.pad;
    a.nby = L.nby;
    a.nbx = L.nbx;
    a.n_ct = L.co_pad / TC_M;
    a.n_chunks = L.ci_pad / TC_CK;
    a.HH = 8 + L.p.k_h - 1;
    a.WW = 8 + L.p.k_w - 1;
    a.taps = L.p.k_h * L.p.k_w;
    a.ci_pad = L.ci_pad;
    a.x5d = L.tc_x5d;
    a.z_tma = (L.y == nullptr && L.tc_z_tma) ? 1 : 0;
    const long long max_units = (long long)L.p.n_streams * L.nby * L.nbx * a.n_ct;
    const int grid = (int)(max_units < L.num_sms ? max_units : L.num_sms);
    conv_tc_kernel<<<grid, TC_THREADS, tc_smem_bytes(a.HH, a.WW), L.stream>>>(tm_xt, L.tmap_xbuf[prev_index],
                                                                              L.tmap_w, L.tmap_z, a);
    return cudaGetLastError();
}

}  // namespace sc
