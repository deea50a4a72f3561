// Warp roles of the weight-stationary tensor-core convolution, shared by the
// stand-alone convolution kernel (sc_conv_ws.cu) and the fused step kernel
// (sc_step_fused.cu).
//
// One CTA owns one weight slice W_s (128 output channels x k*k taps x 64
// input channels) in tensor memory for the whole launch, as the A operand of
// tcgen05.mma, and computes, for each open block it is handed, the slice's
// partial product D_s[co][p] = sum_{tap, c in chunk} W[co][tap][c] r[p+tap][c],
// which the epilogue adds into z~ with a TMA reduce-add (Eq. 3: the slices of
// a block sum into z~ in any order).
//
// The roles are fed by a block queue in shared memory.  The producer writes
// the id of the block it stages into each halo stage (-1 ends the work) and
// the id travels with the stage: residual warps and the MMA warp read it from
// the stage, the MMA warp forwards it to the epilogue with its accumulator.
//
//   producer (1 thread) : x_empty -> stage_blk, TMA halo rows of x_t, x_{t-1} -> x_full
//   residual (4 warps)  : x_full -> r = x_t - x_{t-1} in the canonical layout, written over the
//                         x_{t-1} tile -> r_ready
//   MMA (1 warp)        : acc_empty, r_ready -> k*k*4 MMAs -> commit x_empty, acc_full; acc_blk -> acc_meta
//   epilogue (4 warps)  : acc_meta, acc_full -> TMEM -> acc_empty -> smem staging tile (two in turn
//                         where the kernel has room) -> TMA reduce-add into z~
//
// Every wait is bounded (mbar_wait); a role that gives up raises the CTA's
// abort flag, the others stop at their next wait.
#pragma once

#include "sc_internal.h"
#include "sc_ptx.cuh"
#include "sc_tc_common.cuh"

namespace sc {
namespace ws {

constexpr int MAX_STAGES = 5;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t ACC_COL = 384;   // accumulators at columns 384 and 448
constexpr uint64_t WAIT_NS = 1000000000ull;
constexpr int WBYTES = TC_M * TC_CK * 2;  // one tap of the slice: 128 x 64 bf16

// KS: kernel size (1 or 3); NST: halo stages in flight.
template <int KS, int NST>
struct Geom {
    static constexpr int HH = 8 + KS - 1, WW = 8 + KS - 1, TAPS = KS * KS;
    static constexpr int G = (HH * WW) | 1;                  // odd canonical group stride, 16-byte units
    static constexpr int RB = HH * WW * 128;                 // one staged halo tile (one tensor)
    // stage: x_t, then x_{t-1}, over which r is written (r's canonical layout takes 8 * G 16-byte units)
    static constexpr int SB = ((RB + 8 * G * 16 + 1023) / 1024) * 1024;
    static constexpr int STAGES = NST;
    static constexpr int STAGE_BYTES = NST * SB;
    static constexpr int TAPS_PER_ROUND = STAGE_BYTES / WBYTES;  // weight taps staged per round
    static_assert(NST >= 2 && NST <= MAX_STAGES, "stage count");
    static_assert(TAPS * 32 <= (int)ACC_COL, "slice does not fit in TMEM");
    static_assert(TAPS_PER_ROUND >= 1, "stage area smaller than one weight tap");
};

struct Bars {
    uint64_t x_full[MAX_STAGES], r_ready[MAX_STAGES], x_empty[MAX_STAGES];
    uint64_t acc_full[2], acc_empty[2], acc_meta[2];
    uint64_t w_full, drain;
    uint32_t tmem_base;
    int abort;
    int stage_blk[MAX_STAGES];  // block staged in each halo stage; -1 = end of work
    int acc_blk[2];          // block of each accumulator; -1 = end of work
};
static_assert(sizeof(Bars) <= 256, "barrier block must fit its 256-byte slot");

// A bounded wait whose outcome is the same in every lane of the warp (all
// lanes wait; if any lane gave up, the warp gives up), so that no lane is left
// alone in a warp-collective instruction after an abort.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int* abort, int* err)
{
    const bool ok = ptx::mbar_wait(bar, parity, abort, err, WAIT_NS);
    return __all_sync(0xffffffffu, ok) != 0;
}

// The same across the 128 threads of named barrier `id` (AND-reduction).
__device__ __forceinline__ bool group_wait(int id, uint32_t bar, uint32_t parity, volatile int* abort, int* err)
{
    const bool ok = ptx::mbar_wait(bar, parity, abort, err, WAIT_NS);
    return ptx::named_bar_and(id, 128, ok);
}

// Thread 0, before the first __syncthreads.
__device__ __forceinline__ void init_barriers(Bars* b)
{
    for (int s = 0; s < MAX_STAGES; ++s) {
        ptx::mbar_init(ptx::smem_u32(&b->x_full[s]), 1);
        ptx::mbar_init(ptx::smem_u32(&b->r_ready[s]), 4);
        ptx::mbar_init(ptx::smem_u32(&b->x_empty[s]), 1);
    }
    for (int s = 0; s < 2; ++s) {
        ptx::mbar_init(ptx::smem_u32(&b->acc_full[s]), 1);
        ptx::mbar_init(ptx::smem_u32(&b->acc_empty[s]), 4);
        ptx::mbar_init(ptx::smem_u32(&b->acc_meta[s]), 1);
    }
    ptx::mbar_init(ptx::smem_u32(&b->w_full), 1);
    ptx::mbar_init(ptx::smem_u32(&b->drain), 1);
    b->abort = 0;
    ptx::fence_mbar_init();
}

// Warps 0-3 (tid = 0..127 = output-channel row of the tile): the weight
// slice into TMEM -- lane = row, columns tap*32 .. tap*32+31 = the chunk's 64
// channels as bf16 pairs.  The taps come by TMA (128-byte swizzled rows)
// through the idle stage area, as many per round as it holds; thread 0
// issues, all 128 copy.  Returns false if a round never arrived.
template <int KS, int NST>
__device__ __forceinline__ bool load_weight_slice(const CUtensorMap* tm_w, uint8_t* sX, Bars* b, uint32_t tmem,
                                                  int ci_pad, int chunk, int ct, int tid, volatile int* abort,
                                                  int* err)
{
    using Gm = Geom<KS, NST>;
    const int warp = tid >> 5, row = tid;
    if (tid == 0) ptx::prefetch_tmap(tm_w);
    bool ok = true;
    uint32_t phase = 0;
#pragma unroll 1
    for (int t0 = 0; t0 < Gm::TAPS && ok; t0 += Gm::TAPS_PER_ROUND, phase ^= 1) {
        const int t1 = min(Gm::TAPS, t0 + Gm::TAPS_PER_ROUND);
        if (t0 > 0) ptx::named_bar_sync(1, 128);   // the previous round's taps are read
        if (tid == 0) {
            ptx::mbar_arrive_expect_tx(ptx::smem_u32(&b->w_full), (t1 - t0) * WBYTES);
            for (int t = t0; t < t1; ++t)
                ptx::tma_load_2d(ptx::smem_u32(sX + (t - t0) * WBYTES), tm_w, ptx::smem_u32(&b->w_full),
                                 t * ci_pad + chunk * TC_CK, ct * TC_M);
        }
        ok = group_wait(1, ptx::smem_u32(&b->w_full), phase, abort, err);
        if (!ok) break;
#pragma unroll 1
        for (int t = t0; t < t1; ++t) {
            const uint4* src = (const uint4*)(sX + (t - t0) * WBYTES + row * 128);
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
    }
    ptx::tmem_wait_st();
    return ok;
}

// The producer's side of the block queue (one thread).
template <int KS, int NST>
struct Producer {
    using Gm = Geom<KS, NST>;
    uint8_t* sX;
    Bars* b;
    const CUtensorMap* tm_xt;
    const CUtensorMap* tm_xp;
    volatile int* abort;
    int* err;
    int chunk, pad, nby, nbx;
    int st;
    uint32_t ph, issued, issue_ph;  // issue_ph: bit s = phase of the copy issued into stage s
    bool ok;

    __device__ __forceinline__ void init(uint8_t* sX_, Bars* b_, const CUtensorMap* xt, const CUtensorMap* xp,
                                         volatile int* abort_, int* err_, int chunk_, int pad_, int nby_, int nbx_)
    {
        sX = sX_; b = b_; tm_xt = xt; tm_xp = xp; abort = abort_; err = err_;
        chunk = chunk_; pad = pad_; nby = nby_; nbx = nbx_;
        st = 0; ph = 0; issued = 0; issue_ph = 0; ok = true;
        ptx::prefetch_tmap(tm_xt);
        ptx::prefetch_tmap(tm_xp);
    }

    // Stage the halo rows of open block `id` (both frames, this CTA's channel chunk).
    __device__ __forceinline__ bool push(int id)
    {
        if (!ok) return false;
        int n, by, bx;
        decode_block(id, nby, nbx, n, by, bx);
        const uint32_t xf = ptx::smem_u32(&b->x_full[st]);
        if (!(ok = ptx::mbar_wait(ptx::smem_u32(&b->x_empty[st]), ph ^ 1, abort, err, WAIT_NS))) return false;
        b->stage_blk[st] = id;
        ptx::mbar_arrive_expect_tx(xf, 2 * Gm::RB);
        const uint32_t dst = ptx::smem_u32(sX + st * Gm::SB);
        const int y0 = by * 8 - pad, x0 = bx * 8 - pad;
        ptx::tma_load_4d(dst, tm_xt, xf, chunk * TC_CK, x0, y0, n);
        ptx::tma_load_4d(dst + Gm::RB, tm_xp, xf, chunk * TC_CK, x0, y0, n);
        issue_ph = (issue_ph & ~(1u << st)) | (ph << st);
        issued |= 1u << st;
        if (++st == NST) { st = 0; ph ^= 1; }
        return true;
    }

    // End of work: a stage carrying -1.  After a failure, wait (bounded) for
    // the copies still in flight so that no TMA writes into a finished CTA.
    __device__ __forceinline__ void finish()
    {
        if (ok && (ok = ptx::mbar_wait(ptx::smem_u32(&b->x_empty[st]), ph ^ 1, abort, err, WAIT_NS))) {
            b->stage_blk[st] = -1;
            ptx::mbar_arrive(ptx::smem_u32(&b->x_full[st]));
            return;
        }
        for (int s = 0; s < NST; ++s)
            if (issued & (1u << s))
                ptx::mbar_wait(ptx::smem_u32(&b->x_full[s]), (issue_ph >> s) & 1u, nullptr, nullptr, WAIT_NS);
    }
};

// Residual warps (tid = 0..127): r = x_t - x_{t-1} (bf16) into the no-swizzle
// K-major canonical layout [8-channel group][row][col][8 ch], group stride G,
// written over the x_{t-1} tile: every thread forms its residuals in registers,
// and the four warps meet at named barrier 3 before any of them writes.
template <int KS, int NST>
__device__ __forceinline__ void residual_role(uint8_t* sX, Bars* b, int tid, volatile int* abort, int* err)
{
    using Gm = Geom<KS, NST>;
    const int lane = tid & 31;
    int xs = 0;
    uint32_t xph = 0;
    for (;;) {
        if (!warp_wait(ptx::smem_u32(&b->x_full[xs]), xph, abort, err)) return;
        const int id = b->stage_blk[xs];
        if (id >= 0) {
            const uint4* xt = (const uint4*)(sX + xs * Gm::SB);
            const uint4* xp = (const uint4*)(sX + xs * Gm::SB + Gm::RB);
            uint4* r = (uint4*)(sX + xs * Gm::SB + Gm::RB);
            constexpr int NV = Gm::HH * Gm::WW * 8;  // (pixel, 8-channel group) pairs
            constexpr int PER = (NV + 127) / 128;
            uint4 rv[PER];
#pragma unroll
            for (int u = 0; u < PER; ++u) {
                const int v = tid + 128 * u;
                if (v < NV) rv[u] = bf16x8_sub(xt[v], xp[v]);
            }
            ptx::named_bar_sync(3, 128);
#pragma unroll
            for (int u = 0; u < PER; ++u) {
                const int v = tid + 128 * u;
                if (v < NV) r[(v & 7) * Gm::G + (v >> 3)] = rv[u];
            }
            ptx::fence_proxy_async_smem();
        }
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&b->r_ready[xs]));
        if (id < 0) return;
        if (++xs == NST) { xs = 0; xph ^= 1; }
    }
}

// MMA warp (converged; one elected lane issues): per block, taps x 4 K-steps
// of M=128, N=64, K=16 with A (the slice) from TMEM and B (r) from shared
// memory; each tap is the residual buffer seen from a shifted start.
template <int KS, int NST>
__device__ __forceinline__ void mma_role(uint8_t* sX, Bars* b, uint32_t tmem, volatile int* abort, int* err)
{
    using Gm = Geom<KS, NST>;
    const int lane = threadIdx.x & 31;
    const uint32_t idesc = ptx::idesc_bf16_f32(TC_M, TC_N);
    int xs = 0, acc = 0;
    uint32_t xph = 0, accph = 0;
    bool ok = true, issued = false;
    for (;;) {
        if (!(ok = warp_wait(ptx::smem_u32(&b->acc_empty[acc]), accph ^ 1, abort, err))) break;
        if (!(ok = warp_wait(ptx::smem_u32(&b->r_ready[xs]), xph, abort, err))) break;
        const int id = b->stage_blk[xs];
        if (id < 0) {
            if (lane == 0) {
                b->acc_blk[acc] = -1;
                ptx::mbar_arrive(ptx::smem_u32(&b->acc_meta[acc]));
            }
            __syncwarp();
            break;
        }
        ptx::tc_fence_after();
        const uint32_t d = tmem + ACC_COL + acc * TC_N;
        const uint64_t b0 = ptx::smem_desc(ptx::smem_u32(sX + xs * Gm::SB + Gm::RB), Gm::G * 16, Gm::WW * 16, 0);
        if (ptx::elect_one()) {
#pragma unroll
            for (int t = 0; t < Gm::TAPS; ++t) {
#pragma unroll
                for (int k = 0; k < TC_CK / 16; ++k) {
                    const uint32_t off = (uint32_t)(2 * k * Gm::G + (t / KS) * Gm::WW + (t % KS));  // 16-byte units
                    ptx::mma_bf16_ts(d, tmem + t * 32 + k * 8, b0 + off, idesc, (t | k) != 0);
                }
            }
            ptx::mma_commit(ptx::smem_u32(&b->x_empty[xs]));
            ptx::mma_commit(ptx::smem_u32(&b->acc_full[acc]));
        }
        __syncwarp();
        if (lane == 0) {
            b->acc_blk[acc] = id;
            ptx::mbar_arrive(ptx::smem_u32(&b->acc_meta[acc]));
        }
        __syncwarp();
        issued = true;
        if (++xs == NST) { xs = 0; xph ^= 1; }
        if (++acc == 2) { acc = 0; accph ^= 1; }
    }
    if (!ok && issued) {
        // let the MMAs already issued finish before the CTA releases its memory
        if (ptx::elect_one()) ptx::mma_commit(ptx::smem_u32(&b->drain));
        __syncwarp();
        ptx::mbar_wait(ptx::smem_u32(&b->drain), 0, nullptr, nullptr, WAIT_NS);
    }
}

// Epilogue warps 0-3 (tid = 0..127): accumulator (lane = output channel,
// column = pixel) -> shared memory [pixel][channel] -> TMA reduce-add into
// z~ at (ct*128, bx*8, by*8, n).  With two staging tiles (zbufs = 2) the tile
// of block i is refilled once the reduce-add of block i - 2 has read it, so a
// reduce-add still draining (its z~ lines come from DRAM) does not hold up the
// next block.
__device__ __forceinline__ void epilogue_role(float* sZ, Bars* b, uint32_t tmem, const CUtensorMap* tm_z, int ct,
                                              int nby, int nbx, int tid, volatile int* abort, int* err, int zbufs)
{
    const int warp = tid >> 5, lane = tid & 31;
    int acc = 0, zb = 0;
    uint32_t accph = 0;
    for (;;) {
        if (!group_wait(1, ptx::smem_u32(&b->acc_meta[acc]), accph, abort, err)) break;
        const int id = b->acc_blk[acc];
        if (id < 0) break;
        int n, by, bx;
        decode_block(id, nby, nbx, n, by, bx);
        if (!group_wait(1, ptx::smem_u32(&b->acc_full[acc]), accph, abort, err)) break;
        ptx::tc_fence_after();
        uint32_t r0[32], r1[32];
        const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16) + ACC_COL + acc * TC_N;
        ptx::tmem_ld_32x32b_x32(taddr, r0);
        ptx::tmem_ld_32x32b_x32(taddr + 32, r1);
        ptx::tmem_wait_ld();
        ptx::tc_fence_before();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(ptx::smem_u32(&b->acc_empty[acc]));
        if (++acc == 2) { acc = 0; accph ^= 1; }
        const int col = warp * 32 + lane;
        float* Z = sZ + zb * (TC_N * TC_M);
        if (tid == 0) {
            if (zbufs == 2) ptx::bulk_wait_group_read1();
            else ptx::bulk_wait_group_read0();
        }
        ptx::named_bar_sync(1, 128);
#pragma unroll
        for (int p = 0; p < 32; ++p) {
            Z[p * TC_M + col] = __uint_as_float(r0[p]);
            Z[(p + 32) * TC_M + col] = __uint_as_float(r1[p]);
        }
        ptx::fence_proxy_async_smem();
        ptx::named_bar_sync(1, 128);
        if (tid == 0) {
            ptx::tma_reduce_add_4d(tm_z, ptx::smem_u32(Z), ct * TC_M, bx * 8, by * 8, n);
            ptx::bulk_commit_group();
        }
        if (zbufs == 2) zb ^= 1;
    }
    // the staging tiles must stay valid until the last reduce-add has read them; its writes to z~
    // complete with the grid
    if (tid == 0) ptx::bulk_wait_group_read0();
}

}  // namespace ws
}  // namespace sc
