// Pieces shared by the two tensor-core convolution kernels.
#pragma once

#include "sc_internal.h"

namespace sc {

constexpr int TC_M = 128;   // output channels per MMA tile
constexpr int TC_N = 64;    // output pixels per MMA tile: one 8x8 gate block
constexpr int TC_CK = 64;   // input channels per K chunk
constexpr int TC_ZBYTES = TC_N * TC_M * 4;  // fp32 staging tile of one unit's result

// Bytes of one halo tile (one tensor, one 64-channel chunk) in the no-swizzle
// K-major canonical layout [8-channel group][row][col][8 channels].
__host__ __device__ inline int x_tile_bytes(int HH, int WW) { return 8 * HH * WW * 16; }

// Open-block id -> (stream, block row, block column).
__device__ __forceinline__ void decode_block(int id, int nby, int nbx, int& n, int& by, int& bx)
{
    bx = id % nbx;
    by = (id / nbx) % nby;
    n = id / (nbx * nby);
}

// Eight bf16 residuals x - p, each the bf16 subtraction rounded to nearest
// (packed pairs: four instructions for eight values).
__device__ __forceinline__ uint4 bf16x8_sub(const uint4& x, const uint4& p)
{
    const __nv_bfloat162* a = reinterpret_cast<const __nv_bfloat162*>(&x);
    const __nv_bfloat162* b = reinterpret_cast<const __nv_bfloat162*>(&p);
    uint4 out;
    __nv_bfloat162* o = reinterpret_cast<__nv_bfloat162*>(&out);
#pragma unroll
    for (int k = 0; k < 4; ++k) o[k] = __hsub2(a[k], b[k]);
    return out;
}

// Tensor maps (sc_conv_tc.cu): halo boxes of a frame, and the z state.
bool tc_encode_x_map(CUtensorMap* m, const void* base, const Layer& L, bool five_d);
bool tc_encode_z_map(CUtensorMap* m, const Layer& L);
// Halo rows for the weight-stationary kernels (sc_conv_ws.cu): 4-D boxes of
// 64 channels (128 bytes) x (8+k_w-1) x (8+k_h-1) pixels of one stream.
bool encode_xrow_map(CUtensorMap* m, const void* base, const Layer& L);

}  // namespace sc
