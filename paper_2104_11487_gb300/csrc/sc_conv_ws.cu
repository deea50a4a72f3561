// Weight-stationary tensor-core convolution of the open blocks.
//
// The K dimension (taps x input channels) of the implicit GEMM is split
// into 64-channel chunks and the output channels into 128-row tiles; one
// (output tile, channel chunk) pair is a "slice" of the weights:
//     W_s[co][tap][c],  128 x (k_h*k_w) x 64   (9 taps: 147 KiB)
// Each CTA owns one slice and keeps it in tensor memory for the whole step,
// as the A operand of tcgen05.mma (A read from TMEM costs no shared-memory
// bandwidth, which otherwise caps the tensor core at about 75-80 B/clk of
// operand reads).  It then sweeps its share of the open blocks; per block it
// computes the partial product of its slice
//     D_s[co][p] = sum_{tap, c in chunk} W[co][tap][c] * r[p + tap][c]
// and adds it into z with a TMA reduce-add at L2, so the slices of a block
// sum into z~_t = z~_{t-1} + w * r_t (Eq. 3) in any order.  Weights cross L2
// once per CTA per step instead of once per block.
//
// Halo tiles arrive by TMA as 128-byte pixel rows (64 channels) in a staging
// buffer; the residual warps write r = x_t - x_{t-1} (bf16) into the
// no-swizzle K-major canonical layout [8-channel group][row][col][8 ch] with
// an odd group stride G (16-byte units), free of bank conflicts.  The B
// operand of tap (kh, kw) is that buffer seen from a start shifted by
// (kh*WW + kw)*16 bytes: output rows WW*16 bytes apart, channel groups G*16.
//
// The MMA warp stays converged and one elected lane issues all MMAs of a
// block with compile-time descriptor offsets: issuing from a divergent lane
// with run-time descriptor arithmetic costs about 100-200 cycles per MMA,
// more than the 32-cycle MMA itself.
//
// The kernel is launched as a programmatic dependent of the gate: TMEM
// allocation and the weight load overlap the gate kernel, and the kernel
// waits on the gate's completion only before it reads the open-block list.
//
// Warp roles: 0-3 weight load, then epilogue; 4-7 residual; 8 TMA producer
// (weights once, then halos); 9 TMEM allocation and MMA issue.
#include "sc_internal.h"
#include "sc_ptx.cuh"
#include "sc_tc_common.cuh"

namespace sc {
namespace {

constexpr int WS_XSTAGES = 4;
constexpr int WS_THREADS = 320;
constexpr uint32_t WS_TMEM_COLS = 512;
constexpr uint32_t WS_ACC_COL = 384;   // accumulators at columns 384 and 448
constexpr uint64_t WS_WAIT_NS = 1000000000ull;
constexpr int WS_WBYTES = TC_M * TC_CK * 2;  // one tap of the slice: 128 x 64 bf16

template <int KS>
struct WsGeom {
    static constexpr int HH = 8 + KS - 1, WW = 8 + KS - 1, TAPS = KS * KS;
    static constexpr int G = (HH * WW) | 1;                  // odd canonical group stride, 16-byte units
    static constexpr int RB = HH * WW * 128;                 // one staged halo tile (one tensor)
    static constexpr int SB = ((2 * RB + 8 * G * 16 + 1023) / 1024) * 1024;  // stage: x_t, x_{t-1}, r
    static constexpr size_t SMEM = 1024 + (size_t)WS_XSTAGES * SB + TC_ZBYTES + 256;
    static_assert(TAPS * 32 <= (int)WS_ACC_COL, "slice does not fit in TMEM");
    static_assert(WS_XSTAGES * SB >= TAPS * WS_WBYTES, "stage area too small to stage the weight slice");
};

struct WsArgs {
    const int32_t* list;
    const int32_t* counters;
    int* err;
    int ci_pad, n_chunks, n_slices, pad, nby, nbx;
};

struct WsBars {
    uint64_t x_full[WS_XSTAGES], r_ready[WS_XSTAGES], x_empty[WS_XSTAGES];
    uint64_t acc_full[2], acc_empty[2];
    uint64_t w_full, drain;
    uint32_t tmem_base;
    int abort;
    int n_mine;
};

template <int KS>
__global__ void __launch_bounds__(WS_THREADS, 1)
conv_ws_kernel(const __grid_constant__ CUtensorMap tm_xt, const __grid_constant__ CUtensorMap tm_xp,
               const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_z, const WsArgs a)
{
    using Gm = WsGeom<KS>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sX = smem;
    float* sZ = (float*)(sX + WS_XSTAGES * Gm::SB);
    WsBars* bars = (WsBars*)((uint8_t*)sZ + TC_ZBYTES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int slice = blockIdx.x % a.n_slices;
    const int ct = slice / a.n_chunks, chunk = slice % a.n_chunks;
    const int Q = gridDim.x / a.n_slices, q = blockIdx.x / a.n_slices;

    // ---------------------------------------------------------- prologue
    if (threadIdx.x == 0) {
        for (int s = 0; s < WS_XSTAGES; ++s) {
            ptx::mbar_init(ptx::smem_u32(&bars->x_full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&bars->r_ready[s]), 4);
            ptx::mbar_init(ptx::smem_u32(&bars->x_empty[s]), 1);
        }
        for (int s = 0; s < 2; ++s) {
            ptx::mbar_init(ptx::smem_u32(&bars->acc_full[s]), 1);
            ptx::mbar_init(ptx::smem_u32(&bars->acc_empty[s]), 4);
        }
        ptx::mbar_init(ptx::smem_u32(&bars->w_full), 1);
        ptx::mbar_init(ptx::smem_u32(&bars->drain), 1);
        bars->abort = 0;
        ptx::fence_mbar_init();
    }
    if (warp == 9) {
        ptx::tmem_alloc(ptx::smem_u32(&bars->tmem_base), WS_TMEM_COLS);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort = &bars->abort;

    // The weight slice: one TMA burst into the (still idle) stage area,
    // 128-byte swizzled rows, then into TMEM: lane = output channel within
    // the tile, columns tap*32 .. tap*32+31 = the chunk's 64 channels as
    // bf16 pairs.
    if (warp == 8 && lane == 0) {
        ptx::prefetch_tmap(&tm_w);
        ptx::mbar_arrive_expect_tx(ptx::smem_u32(&bars->w_full), Gm::TAPS * WS_WBYTES);
        for (int t = 0; t < Gm::TAPS; ++t)
            ptx::tma_load_2d(ptx::smem_u32(sX + t * WS_WBYTES), &tm_w, ptx::smem_u32(&bars->w_full),
                             t * a.ci_pad + chunk * TC_CK, ct * TC_M);
    }
    bool w_ok = true;
    if (warp < 4) {
        w_ok = ptx::mbar_wait(ptx::smem_u32(&bars->w_full), 0, abort, a.err, WS_WAIT_NS);
        if (w_ok) {
            const int row = threadIdx.x;
#pragma unroll 1
            for (int t = 0; t < Gm::TAPS; ++t) {
                const uint4* src = (const uint4*)(sX + t * WS_WBYTES + row * 128);
                uint32_t v[32];
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    const uint4 u = src[c ^ (row & 7)];   // 128-byte swizzle: chunk c of row r sits at c ^ (r % 8)
                    v[4 * c] = u.x;
                    v[4 * c + 1] = u.y;
                    v[4 * c + 2] = u.z;
                    v[4 * c + 3] = u.w;
                }
                ptx::tmem_st_32x32b_x32(tmem + ((uint32_t)(warp * 32) << 16) + t * 32, v);
            }
            ptx::tmem_wait_st();
        }
    }
    // The open-block list is written by the gate kernel this grid depends on.
    ptx::grid_dependency_wait();
    if (threadIdx.x == 0) {
        const int count = a.counters[0];
        bars->n_mine = count > q ? (count - q + Q - 1) / Q : 0;  // open blocks q, q+Q, ...
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const int n_mine = w_ok && !*abort ? bars->n_mine : 0;

    if (warp == 8) {
        // --------------------------------------------- halo producer
        if (lane == 0) {
            ptx::prefetch_tmap(&tm_xt);
            ptx::prefetch_tmap(&tm_xp);
            int st = 0;
            uint32_t ph = 0, issue_ph[WS_XSTAGES] = {}, issued = 0;
            bool ok = true;
            for (int i = 0; i < n_mine && ok; ++i) {
                int n, by, bx;
                decode_block(a.list[q + i * Q], a.nby, a.nbx, n, by, bx);
                const int y0 = by * 8 - a.pad, x0 = bx * 8 - a.pad;
                const uint32_t xf = ptx::smem_u32(&bars->x_full[st]);
                if (!(ok = ptx::mbar_wait(ptx::smem_u32(&bars->x_empty[st]), ph ^ 1, abort, a.err, WS_WAIT_NS)))
                    break;
                ptx::mbar_arrive_expect_tx(xf, 2 * Gm::RB);
                const uint32_t dst = ptx::smem_u32(sX + st * Gm::SB);
                ptx::tma_load_4d(dst, &tm_xt, xf, chunk * TC_CK, x0, y0, n);
                ptx::tma_load_4d(dst + Gm::RB, &tm_xp, xf, chunk * TC_CK, x0, y0, n);
                issue_ph[st] = ph;
                issued |= 1u << st;
                if (++st == WS_XSTAGES) { st = 0; ph ^= 1; }
            }
            if (!ok) {
                for (int s = 0; s < WS_XSTAGES; ++s)
                    if (issued & (1u << s))
                        ptx::mbar_wait(ptx::smem_u32(&bars->x_full[s]), issue_ph[s], nullptr, nullptr, WS_WAIT_NS);
            }
        }
    } else if (warp == 9) {
        // ------------------------------- MMA issue (converged warp, one elected lane)
        const uint32_t idesc = ptx::idesc_bf16_f32(TC_M, TC_N);
        int xs = 0, acc = 0;
        uint32_t xph = 0, accph = 0;
        bool ok = true, issued = false;
        for (int i = 0; i < n_mine && ok; ++i) {
            if (!(ok = ptx::mbar_wait(ptx::smem_u32(&bars->acc_empty[acc]), accph ^ 1, abort, a.err, WS_WAIT_NS)))
                break;
            if (!(ok = ptx::mbar_wait(ptx::smem_u32(&bars->r_ready[xs]), xph, abort, a.err, WS_WAIT_NS))) break;
            ptx::tc_fence_after();
            const uint32_t d = tmem + WS_ACC_COL + acc * TC_N;
            const uint64_t b0 = ptx::smem_desc(ptx::smem_u32(sX + xs * Gm::SB + 2 * Gm::RB), Gm::G * 16, Gm::WW * 16, 0);
            if (ptx::elect_one()) {
#pragma unroll
                for (int t = 0; t < Gm::TAPS; ++t) {
#pragma unroll
                    for (int k = 0; k < TC_CK / 16; ++k) {
                        const uint32_t off = (uint32_t)(2 * k * Gm::G + (t / KS) * Gm::WW + (t % KS));  // 16-byte units
                        ptx::mma_bf16_ts(d, tmem + t * 32 + k * 8, b0 + off, idesc, (t | k) != 0);
                    }
                }
                ptx::mma_commit(ptx::smem_u32(&bars->x_empty[xs]));
                ptx::mma_commit(ptx::smem_u32(&bars->acc_full[acc]));
            }
            __syncwarp();
            issued = true;
            if (++xs == WS_XSTAGES) { xs = 0; xph ^= 1; }
            if (++acc == 2) { acc = 0; accph ^= 1; }
        }
        if (!ok && issued) {
            if (ptx::elect_one()) ptx::mma_commit(ptx::smem_u32(&bars->drain));
            __syncwarp();
            ptx::mbar_wait(ptx::smem_u32(&bars->drain), 0, nullptr, nullptr, WS_WAIT_NS);
        }
    } else if (warp >= 4) {
        // --------------------------------- residual r = x_t - x_{t-1}
        const int tid = threadIdx.x - 128;
        int xs = 0;
        uint32_t xph = 0;
        for (int i = 0; i < n_mine; ++i) {
            if (!ptx::mbar_wait(ptx::smem_u32(&bars->x_full[xs]), xph, abort, a.err, WS_WAIT_NS)) break;
            const uint4* xt = (const uint4*)(sX + xs * Gm::SB);
            const uint4* xp = (const uint4*)(sX + xs * Gm::SB + Gm::RB);
            uint4* r = (uint4*)(sX + xs * Gm::SB + 2 * Gm::RB);
            constexpr int NV = Gm::HH * Gm::WW * 8;  // (pixel, 8-channel group) pairs
#pragma unroll 4
            for (int v = tid; v < NV; v += 128) r[(v & 7) * Gm::G + (v >> 3)] = bf16x8_sub(xt[v], xp[v]);
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&bars->r_ready[xs]));
            if (++xs == WS_XSTAGES) { xs = 0; xph ^= 1; }
        }
    } else {
        // ------------------------ epilogue: z += D_s (TMA reduce-add)
        const int tid = threadIdx.x;
        int acc = 0;
        uint32_t accph = 0;
        for (int i = 0; i < n_mine; ++i) {
            int n, by, bx;
            decode_block(a.list[q + i * Q], a.nby, a.nbx, n, by, bx);
            if (!ptx::mbar_wait(ptx::smem_u32(&bars->acc_full[acc]), accph, abort, a.err, WS_WAIT_NS)) break;
            ptx::tc_fence_after();
            uint32_t r0[32], r1[32];
            const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + WS_ACC_COL + acc * TC_N;
            ptx::tmem_ld_32x32b_x32(taddr, r0);
            ptx::tmem_ld_32x32b_x32(taddr + 32, r1);
            ptx::tmem_wait_ld();
            ptx::tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&bars->acc_empty[acc]));
            if (++acc == 2) { acc = 0; accph ^= 1; }
            const int col = warp * 32 + lane;
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
        }
        if (tid == 0) ptx::bulk_wait_group0();
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        __syncwarp();
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, WS_TMEM_COLS);
    }
}

// Halo boxes of 64 channels (128-byte rows) x (8+k_w-1) x (8+k_h-1) pixels.
bool encode_xrow_map(CUtensorMap* m, const void* base, const Layer& L)
{
    EncodeTiledFn enc = encode_tiled_fn();
    if (!enc) return false;
    const cuuint64_t C = L.p.c_in, W = L.p.w, H = L.p.h, N = L.p.n_streams;
    cuuint64_t dims[4] = {C, W, H, N};
    cuuint64_t strides[3] = {C * 2, W * C * 2, H * W * C * 2};
    cuuint32_t box[4] = {TC_CK, (cuuint32_t)(8 + L.p.k_w - 1), (cuuint32_t)(8 + L.p.k_h - 1), 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int KS>
cudaError_t launch_ks(const Layer& L, const CUtensorMap& tm_xt, int prev_index, const WsArgs& a, int grid)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(WS_THREADS);
    cfg.dynamicSmemBytes = WsGeom<KS>::SMEM;
    cfg.stream = L.stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, conv_ws_kernel<KS>, tm_xt, L.tmap_xrow[prev_index], L.tmap_w, L.tmap_z, a);
}

}  // namespace

bool conv_ws_supported(const Layer& L)
{
    return L.path == SKIPCONV_PATH_TENSOR_CORE && L.y == nullptr && L.tc_z_tma && L.p.k_h == L.p.k_w &&
           (L.p.k_h == 1 || L.p.k_h == 3);
}

cudaError_t conv_ws_prepare(Layer& L)
{
    if (!encode_xrow_map(&L.tmap_xrow[0], L.xbuf[0], L) || !encode_xrow_map(&L.tmap_xrow[1], L.xbuf[1], L)) {
        set_error("tensor map of the state frames rejected");
        return cudaErrorInvalidValue;
    }
    if (L.p.k_h == 3)
        return cudaFuncSetAttribute(conv_ws_kernel<3>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)WsGeom<3>::SMEM);
    return cudaFuncSetAttribute(conv_ws_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)WsGeom<1>::SMEM);
}

cudaError_t launch_conv_ws(const Layer& L, const void* x_t, int prev_index)
{
    alignas(64) CUtensorMap tm_xt;
    if (!encode_xrow_map(&tm_xt, x_t, L)) {
        set_error("tensor map of x_t rejected");
        return cudaErrorInvalidValue;
    }
    WsArgs a;
    a.list = L.list;
    a.counters = step_count(L);
    a.err = L.err_dev;
    a.ci_pad = L.ci_pad;
    a.n_chunks = L.ci_pad / TC_CK;
    a.n_slices = (L.co_pad / TC_M) * a.n_chunks;
    a.pad = L.p.pad;
    a.nby = L.nby;
    a.nbx = L.nbx;
    const int per_slice = L.num_sms / a.n_slices > 0 ? L.num_sms / a.n_slices : 1;
    const int grid = a.n_slices * per_slice;
    return L.p.k_h == 3 ? launch_ks<3>(L, tm_xt, prev_index, a, grid) : launch_ks<1>(L, tm_xt, prev_index, a, grid);
}

}  // namespace sc
