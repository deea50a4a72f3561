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
#include "sc_ws_roles.cuh"

namespace sc {
namespace {

constexpr int WS_THREADS = 320;
constexpr int WS_STAGES = 4;

template <int KS>
constexpr size_t ws_smem_bytes() { return 1024 + (size_t)ws::Geom<KS, WS_STAGES>::STAGE_BYTES + 2 * TC_ZBYTES + 256; }

struct WsArgs {
    const int32_t* list;
    const int32_t* counters;
    int* err;
    int ci_pad, n_chunks, n_slices, pad, nby, nbx;
};

template <int KS>
__global__ void __launch_bounds__(WS_THREADS, 1)
conv_ws_kernel(const __grid_constant__ CUtensorMap tm_xt, const __grid_constant__ CUtensorMap tm_xp,
               const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_z, const WsArgs a)
{
    using Gm = ws::Geom<KS, WS_STAGES>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = ptx::align_smem_1024(smem_raw);
    uint8_t* sX = smem;
    float* sZ = (float*)(sX + Gm::STAGE_BYTES);
    ws::Bars* bars = (ws::Bars*)((uint8_t*)sZ + 2 * TC_ZBYTES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int slice = blockIdx.x % a.n_slices;
    const int ct = slice / a.n_chunks, chunk = slice % a.n_chunks;
    const int Q = gridDim.x / a.n_slices, q = blockIdx.x / a.n_slices;

    if (threadIdx.x == 0) ws::init_barriers(bars);
    if (warp == 9) {
        ptx::tmem_alloc(ptx::smem_u32(&bars->tmem_base), ws::TMEM_COLS);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort = &bars->abort;

    if (warp < 4)
        ws::load_weight_slice<KS, WS_STAGES>(&tm_w, sX, bars, tmem, a.ci_pad, chunk, ct, threadIdx.x, abort, a.err);
    // the stage area held the slice: every role starts after the copy into TMEM
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();

    if (warp == 8) {
        if (lane == 0) {
            ws::Producer<KS, WS_STAGES> pr;
            pr.init(sX, bars, &tm_xt, &tm_xp, abort, a.err, chunk, a.pad, a.nby, a.nbx);
            // The open-block list is written by the gate kernel this grid depends on.
            ptx::grid_dependency_wait();
            const int count = *abort ? 0 : a.counters[0];
            for (int e = q; e < count; e += Q)
                if (!pr.push(a.list[e])) break;
            pr.finish();
        }
    } else if (warp == 9) {
        ws::mma_role<KS, WS_STAGES>(sX, bars, tmem, abort, a.err);
    } else if (warp >= 4) {
        ws::residual_role<KS, WS_STAGES>(sX, bars, threadIdx.x - 128, abort, a.err);
    } else {
        ws::epilogue_role(sZ, bars, tmem, &tm_z, ct, a.nby, a.nbx, threadIdx.x, abort, a.err, 2);
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        __syncwarp();
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, ws::TMEM_COLS);
    }
}

template <int KS>
cudaError_t launch_ks(const Layer& L, const CUtensorMap& tm_xt, int prev_index, const WsArgs& a, int grid)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(WS_THREADS);
    cfg.dynamicSmemBytes = ws_smem_bytes<KS>();
    cfg.stream = L.stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, conv_ws_kernel<KS>, tm_xt, L.tmap_xrow[prev_index], L.tmap_w, L.tmap_z, a);
}

}  // namespace

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
                                    (int)ws_smem_bytes<3>());
    return cudaFuncSetAttribute(conv_ws_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)ws_smem_bytes<1>());
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
