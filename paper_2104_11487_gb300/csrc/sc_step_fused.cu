// The whole Skip-Conv step in one persistent launch (one CTA per SM,
// cooperative launch so that all CTAs are resident together).
//
// The three parts of the step -- the per-pixel residual norm and state commit
// (gate pass 1), the block gate (pass 2) and the convolution of the open
// blocks (Eq. 3) -- run concurrently in different warps of every CTA and are
// pipelined over the independent streams n = 0, 1, ...:
//
//   gate warps (8, or fewer in the busier launch forms below)
//       stream this CTA's share of every stream's pixels, in stream order,
//       through shared-memory slots that each warp refills by bulk copies (no
//       registers or L1 held by loads in flight); form r_t = x_t - x_{t-1}
//       (Eq. 2) and its channel l1 norm (Eq. 5), publish the norm, commit x_t
//       where it changed;
//   2 block-gate warps (streams of even / odd n)
//       evaluate this CTA's share of each stream's gate blocks (support sums
//       of the norms over the block's footprint, block max, threshold; Eq. 5
//       and Sec. 3.2) as soon as the footprint's norms are published, and
//       publish the gate decision;
//   convolution (sc_ws_roles.cuh)
//       the producer warp waits for stream n's gate decisions, deals the open
//       blocks of the step round-robin over the CTAs of its weight slice and
//       feeds them to the weight-stationary roles, which add the slice's
//       partial products into z~ (TMA reduce-add).
//
// So the convolution of stream n overlaps the streaming of the streams after
// it and reads its halo rows while they are still in L2.  The kernel is
// instantiated in three forms that split the shared memory differently
// between the gate's ring slots and the convolution's halo stages (FsCfg
// below): the sparse form, a form for steps expected to open many blocks,
// and a form for forced steps.
//
// Hand-off between CTAs carries its own readiness: a published norm is one
// 64-bit word (step epoch, fp32 norm) and a gate decision one 32-bit word
// (step epoch, open bit), each written with a relaxed max reduction at L2 and
// read with single-copy-atomic relaxed loads; a reader polls the words it needs
// until all carry this step's epoch.  Every step rewrites every word, so no
// counter or fence is needed (the words are cleared only before the epoch
// wraps around), and each hop costs one memory round trip.  Every CTA
// derives the same ordered list of open blocks from the decisions, so no
// atomics build it; the CTA that owns stream n (n mod grid) writes that
// stream's part of the ABI's list.  Every poll is bounded; a CTA that gives
// up raises a grid-wide abort flag.
#include "sc_internal.h"
#include "sc_ws_roles.cuh"

namespace sc {
namespace {

constexpr int FS_MAX_GATE_WARPS = 8;              // gate warps of the widest form (barrier slots)
constexpr int FS_BG_WARPS = 2;                     // block-gate warps

// Warp roles per CTA: 0-3 epilogue, 4-7 residual, 8 producer, 9 MMA, 10-11
// block gate, 12.. gate.  NG gate warps (= ring slots), NST halo stages.
// A sparse step streams with 8 gate warps and 3 halo stages.  When the last
// sparse step opened at least 3/8 of the blocks, the convolution is most of
// the work and 6 gate warps / 4 halo stages pay instead (c4, us per step at
// 10 / 25 / 50 / 100 % density: 8 / 3 43.2, 55.2, 82.1, 132.7; 6 / 4 49.5,
// 57.8, 79.9, 125.7).  In a forced step (key frame, dense mode) every
// decision is published at once, so the convolution starts at the kernel's
// start; the gate only commits x_t beside it, which 2 gate warps finish well
// before the convolution does, and the six ring slots this frees buy two more
// halo stages (a dense c4 step: 8 / 3 129.0 us, 6 / 4 123.5, 3 / 5 120.3,
// 2 / 5 118.1, 4 / 4 124.1).
template <int NG, int NST>
struct FsCfg {
    static constexpr int GATE_WARPS = NG, STAGES = NST;
    static constexpr int WARPS = 10 + FS_BG_WARPS + NG;
    static constexpr int THREADS = WARPS * 32;
    static_assert(NG <= FS_MAX_GATE_WARPS, "gate warps");
};
using CfgSparse = FsCfg<8, 3>;
using CfgBusy = FsCfg<6, 4>;
using CfgForced = FsCfg<2, 5>;
constexpr int FS_SLOT = 8192;                      // ring slot: x_t chunk | x_{t-1} chunk
constexpr int FS_HALF = FS_SLOT / 2;
constexpr int FS_FOOT = 16 * 16;                   // block-gate footprint capacity (floats)

struct FusedArgs {
    // gate pass 1
    const uint8_t* xt;
    const uint8_t* xp;
    uint4* xn;
    const uint8_t* chg_prev;
    uint8_t* chg_cur;
    uint64_t* pnorm;       // per pixel: (epoch << 32) | fp32 l1 norm of r
    int n, P, W, H, units, log2g, pb, gch;   // pb: bytes per pixel; gch: pixels per ring chunk
    // gate pass 2
    uint8_t* mask;
    uint32_t* gtag;        // per gate block: (epoch << 1) | open
    int32_t* list;
    int32_t* count;        // this step's open-block count (the ABI's view)
    int* hint;             // mapped host word: this step's open-block count (sparse steps), a launch hint
    int* gabort;           // grid-wide abort flag
    uint32_t epoch;        // this step's tag, 1 .. 2^31 - 1
    float thr;
    int force;
    int Ho, Wo, KH, KW, pad, nby, nbx;
    // convolution
    int* err;
    int ci_pad, n_chunks, n_slices;
};

struct FusedShared {
    uint64_t g_full[FS_MAX_GATE_WARPS];
    float foot[FS_BG_WARPS][2][FS_FOOT];   // block-gate footprints of pixel norms
};

template <int KS, class C>
constexpr size_t fused_smem_bytes()
{
    return 1024 + (size_t)ws::Geom<KS, C::STAGES>::STAGE_BYTES + (size_t)C::GATE_WARPS * FS_SLOT + 2 * TC_ZBYTES +
           256 + sizeof(FusedShared);
}

__device__ __forceinline__ uint64_t ld_relaxed_u64(const uint64_t* p)
{
    uint64_t v;
    asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ uint32_t ld_relaxed_u32(const uint32_t* p)
{
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Publish a tagged word for pollers on other SMs: a relaxed max reduction,
// performed at the word's home in L2, so a poller on either die sees it after
// one round trip (a plain store was measured to linger for microseconds before
// other SMs observed it).  The step epoch sits in the high bits and only grows
// between resets of the words, so the maximum is the new word.  A reduction
// returns nothing: the writing warp does not wait for the round trip.
__device__ __forceinline__ void publish_u64(uint64_t* p, uint64_t v)
{
    asm volatile("red.relaxed.gpu.global.max.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ void publish_u32(uint32_t* p, uint32_t v)
{
    asm volatile("red.relaxed.gpu.global.max.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ uint4 ld_relaxed_v4(const uint32_t* p)
{
    uint4 v;
    asm volatile("ld.relaxed.gpu.global.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p)
                 : "memory");
    return v;
}

// Between two polls of a warp that waits for published words: give up (false,
// the same in every lane) after the time limit or once any CTA raised the
// abort flag.  `gab` is lane 0's copy of the grid abort flag, loaded together
// with the polled words.  There is no sleep between polls: each poll is
// already one memory round trip, and a sleep only delays seeing the last word.
__device__ __forceinline__ bool keep_polling(uint64_t t0, int gab, const FusedArgs& a, volatile int* abort, int lane)
{
    int give_up = 0;
    if (lane == 0) {
        if (gab || *abort) {
            give_up = 1;
        } else if (ptx::globaltimer() - t0 > ws::WAIT_NS) {
            *(volatile int*)a.err = DEV_TIMEOUT;
            atomicExch(a.gabort, 1);
            give_up = 1;
        }
        if (give_up) *abort = 1;
    }
    give_up = __shfl_sync(0xffffffffu, give_up, 0);
    return give_up == 0;
}

__device__ __forceinline__ int ld_relaxed_i32(const int* p)
{
    int v;
    asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ float l1_bf16x8(const uint4& a, const uint4& b)
{
    const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
    const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b);
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 fa = __bfloat1622float2(pa[k]);
        const float2 fb = __bfloat1622float2(pb[k]);
        s += fabsf(fa.x - fb.x) + fabsf(fa.y - fb.y);
    }
    return s;
}

// This CTA's pixels of every stream: [lo, hi) of each stream's h*w, cut into
// chunks of gch pixels; chunk k (stream n = k / cpn) goes to ring slot and
// gate warp k % NG.
struct GateRange {
    int lo, hi, cpn, total;
    __device__ __forceinline__ GateRange(const FusedArgs& a)
    {
        lo = (int)((long long)blockIdx.x * a.P / gridDim.x);
        hi = (int)((long long)(blockIdx.x + 1) * a.P / gridDim.x);
        cpn = (hi - lo + a.gch - 1) / a.gch;
        total = a.n * cpn;
    }
};

// Gate warp gw: chunks gw, gw + 8, ... through ring slot gw, which the warp
// refills itself (lane 0, two bulk copies: the chunk of x_t and of x_{t-1})
// as soon as it has read the previous chunk into registers -- eight issuing
// threads per SM keep enough copies in flight to stream at full bandwidth.
// A chunk is 8 rows of 32 / G pixels, G = 2^LOG2G lanes per pixel (one
// 16-byte unit each).  The 8 per-lane sums are reduced over the pixel's G
// lanes by a transposed butterfly: three halving exchanges leave one row's
// sum in each lane (row index = the lane's top three sub-lane bits), then
// plain steps; the pairing is that of a plain xor butterfly, so the sums are
// bit-identical to it.
template <int LOG2G, int NG>
__device__ void gate_pixels_role(const FusedArgs& a, FusedShared* sh, const uint8_t* ring, int gw, int lane,
                                 volatile int* abort)
{
    constexpr int G = 1 << LOG2G, ROWS = 32 >> LOG2G, CH = 8 * ROWS;
    static_assert(LOG2G >= 3 && LOG2G <= 5, "8 to 32 lanes per pixel");
    const GateRange R(a);
    if (R.cpn == 0) return;
    const int sub = lane & (G - 1), prow = lane >> LOG2G;
    const bool lane_on = sub < a.units;
    const uint4* sxt = (const uint4*)(ring + gw * FS_SLOT);
    const uint4* sxp = (const uint4*)(ring + gw * FS_SLOT + FS_HALF);
    const uint32_t full = ptx::smem_u32(&sh->g_full[gw]);
    // lane 0: chunk k of this CTA's share into the slot
    auto issue = [&](int k) {
        const int n = k / R.cpn;
        const int p0 = R.lo + (k - n * R.cpn) * CH;
        const uint32_t bytes = (uint32_t)(min(CH, R.hi - p0) * a.pb);
        const size_t off = ((size_t)n * a.P + p0) * a.pb;
        ptx::mbar_arrive_expect_tx(full, 2 * bytes);
        ptx::bulk_load(ptx::smem_u32(ring + gw * FS_SLOT), a.xt + off, bytes, full);
        ptx::bulk_load(ptx::smem_u32(ring + gw * FS_SLOT + FS_HALF), a.xp + off, bytes, full);
    };
    // the previous step's change flag of pixel `lane` of chunk k (<= 32 pixels), loaded one chunk ahead
    auto chg_of = [&](int k) -> uint32_t {
        const int n = k / R.cpn;
        const int p0 = R.lo + (k - n * R.cpn) * CH;
        return (k < R.total && lane < min(CH, R.hi - p0)) ? a.chg_prev[(long long)n * a.P + p0 + lane] : 0u;
    };
    if (lane == 0 && gw < R.total) issue(gw);
    uint32_t chg_next = chg_of(gw);
    // the row whose sum this lane holds after the halving exchanges
    const int my_row = (((sub >> (LOG2G - 1)) & 1) << 2) | (((sub >> (LOG2G - 2)) & 1) << 1) | ((sub >> (LOG2G - 3)) & 1);
    const bool writer = (sub & ((G >> 3) - 1)) == 0;
    uint32_t ph = 0;
    for (int k = gw; k < R.total; k += NG, ph ^= 1u) {
        const int n = k / R.cpn;
        const int p0 = R.lo + (k - n * R.cpn) * CH;
        const int np = min(CH, R.hi - p0);
        const long long base = (long long)n * a.P + p0;
        const uint32_t cm = __ballot_sync(0xffffffffu, chg_next != 0);
        chg_next = chg_of(k + NG);
        if (!ws::warp_wait(full, ph, abort, a.err)) {
            // the copy in flight may still land: wait for it (bounded) before the CTA can exit
            if (lane == 0) ptx::mbar_wait(full, ph, nullptr, nullptr, ws::WAIT_NS);
            return;
        }
        uint4 av[8];
        float s[8];
        uint32_t d[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int i = u * ROWS + prow;
            uint4 b = make_uint4(0, 0, 0, 0);
            av[u] = b;
            if (i < np && lane_on) {
                av[u] = sxt[i * a.units + sub];
                b = sxp[i * a.units + sub];
            }
            s[u] = l1_bf16x8(av[u], b);
            d[u] = (av[u].x ^ b.x) | (av[u].y ^ b.y) | (av[u].z ^ b.z) | (av[u].w ^ b.w);
        }
        __syncwarp();
        if (lane == 0 && k + NG < R.total) {
            ptx::fence_proxy_async_smem();   // the slot's reads before the copy that overwrites it
            issue(k + NG);
        }
        // transposed butterfly over the pixel's G lanes
        float t4[4], t2[2], t1;
        {
            const bool h = (sub >> (LOG2G - 1)) & 1;
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const float send = h ? s[r] : s[r + 4], keep = h ? s[r + 4] : s[r];
                t4[r] = keep + __shfl_xor_sync(0xffffffffu, send, G >> 1);
            }
        }
        {
            const bool h = (sub >> (LOG2G - 2)) & 1;
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                const float send = h ? t4[r] : t4[r + 2], keep = h ? t4[r + 2] : t4[r];
                t2[r] = keep + __shfl_xor_sync(0xffffffffu, send, G >> 2);
            }
        }
        {
            const bool h = (sub >> (LOG2G - 3)) & 1;
            const float send = h ? t2[0] : t2[1], keep = h ? t2[1] : t2[0];
            t1 = keep + __shfl_xor_sync(0xffffffffu, send, G >> 3);
        }
#pragma unroll
        for (int off = (G >> 4); off > 0; off >>= 1) t1 += __shfl_xor_sync(0xffffffffu, t1, off);
        // changed pixels: any lane of the pixel's group saw a bit difference
        uint32_t chg_rows = 0;   // bit u: row u of this lane's pixel column changed
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const uint32_t bal = __ballot_sync(0xffffffffu, d[u] != 0);
            const uint32_t grp = G == 32 ? bal : (bal >> (prow * G)) & ((1u << G) - 1u);
            chg_rows |= (grp != 0 ? 1u : 0u) << u;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            const int i = u * ROWS + prow;
            if (i < np && lane_on && (((chg_rows >> u) & 1u) || ((cm >> i) & 1u)))
                a.xn[(base + i) * a.units + sub] = av[u];
        }
        {
            const int i = my_row * ROWS + prow;
            if (writer && i < np) {
                publish_u64(a.pnorm + base + i, ((uint64_t)a.epoch << 32) | __float_as_uint(t1));
                a.chg_cur[base + i] = (chg_rows >> my_row) & 1u;
            }
        }
    }
}

// Gate pass 2, block-gate warp wb: streams n = wb, wb + 2, ..., and for each
// this CTA's share of its gate blocks (j = blockIdx.x, blockIdx.x + grid, ...),
// two blocks per round.  The footprint of a block's 8x8 outputs (stride 1) is
// (7+KS) x (7+KS) pixels; its norms are polled until every word carries this
// step's epoch, then each lane sums the KS x KS supports of two outputs.
template <int KS>
__device__ void gate_blocks_role(const FusedArgs& a, FusedShared* sh, volatile int* abort, int wb, int lane)
{
    constexpr int FW = 7 + KS, FF = FW * FW, R = (FF + 31) / 32;
    static_assert(FF <= FS_FOOT, "footprint");
    const int nb = a.nby * a.nbx;
    float(*foot)[FS_FOOT] = sh->foot[wb];
    for (int n = wb; n < a.n; n += FS_BG_WARPS) {
        const uint64_t* Pn = a.pnorm + (size_t)n * a.P;
        for (int j0 = blockIdx.x; j0 < nb; j0 += 2 * gridDim.x) {
            int open[2] = {1, 1};
            if (!a.force) {
                uint64_t v[2][R];
                const uint64_t* src[2][R];
                uint32_t need = 0;   // bit u*R + r: an in-frame footprint word not yet seen with this epoch
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int j = j0 + u * gridDim.x;
                    const int by = j / a.nbx, bx = j - by * a.nbx;
                    const int fy0 = by * 8 - a.pad, fx0 = bx * 8 - a.pad;
#pragma unroll
                    for (int r = 0; r < R; ++r) {
                        const int q = lane + 32 * r;
                        const int yy = fy0 + q / FW, xx = fx0 + q % FW;
                        v[u][r] = 0;
                        src[u][r] = Pn + (size_t)yy * a.W + xx;
                        if (j < nb && q < FF && yy >= 0 && yy < a.H && xx >= 0 && xx < a.W) need |= 1u << (u * R + r);
                    }
                }
                const uint64_t t0 = ptx::globaltimer();
                bool ok = true;
                for (;;) {
                    const int gab = lane == 0 ? ld_relaxed_i32(a.gabort) : 0;
#pragma unroll
                    for (int u = 0; u < 2; ++u)
#pragma unroll
                        for (int r = 0; r < R; ++r)
                            if ((need >> (u * R + r)) & 1u) v[u][r] = ld_relaxed_u64(src[u][r]);
#pragma unroll
                    for (int u = 0; u < 2; ++u)
#pragma unroll
                        for (int r = 0; r < R; ++r)
                            if ((uint32_t)(v[u][r] >> 32) == a.epoch) need &= ~(1u << (u * R + r));
                    if (!__any_sync(0xffffffffu, need != 0)) break;
                    if (!(ok = keep_polling(t0, gab, a, abort, lane))) break;
                }
                if (!ok) return;
#pragma unroll
                for (int u = 0; u < 2; ++u)
#pragma unroll
                    for (int r = 0; r < R; ++r)
                        if (lane + 32 * r < FF) foot[u][lane + 32 * r] = __uint_as_float((uint32_t)v[u][r]);
                __syncwarp();
                // outputs (i, jj) = (lane / 8, lane % 8) and (lane / 8 + 4, lane % 8)
                const int oi = lane >> 3, oj = lane & 7;
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int j = j0 + u * gridDim.x;
                    const int by = j / a.nbx, bx = j - by * a.nbx;
                    const int bh = min(8, a.Ho - by * 8), bw = min(8, a.Wo - bx * 8);
                    float best = -1.f;
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int i = oi + 4 * h;
                        float S = 0.f;
#pragma unroll
                        for (int kh = 0; kh < KS; ++kh)
#pragma unroll
                            for (int kw = 0; kw < KS; ++kw) S += foot[u][(i + kh) * FW + oj + kw];
                        if (i < bh && oj < bw) best = fmaxf(best, S);
                    }
#pragma unroll
                    for (int off = 16; off > 0; off >>= 1)
                        best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, off));
                    open[u] = best > a.thr ? 1 : 0;
                }
                __syncwarp();
            }
            if (lane < 2) {
                const int j = j0 + lane * gridDim.x;
                if (j < nb) {
                    a.mask[(size_t)n * nb + j] = (uint8_t)open[lane];
                    publish_u32(a.gtag + (size_t)n * nb + j, (a.epoch << 1) | (uint32_t)open[lane]);
                }
            }
        }
    }
}

template <int KS, int NST>
__device__ void conv_producer_role(const FusedArgs& a, ws::Producer<KS, NST>& pr, bool conv_cta, int Q, int q,
                                   volatile int* abort, int lane)
{
    const int nb = a.nby * a.nbx;
    int gprefix = 0;
    bool ok = true;
    for (int n = 0; n < a.n && ok; ++n) {
        const uint32_t* trow = a.gtag + (size_t)n * nb;
        const bool owner = (int)blockIdx.x == n % (int)gridDim.x;
        for (int base = 0; base < nb && ok; base += 256) {
            const int j0 = base + lane * 8;
            // this lane's 8 gate decisions, polled until all carry this step's epoch
            uint32_t w[8];
            uint32_t need = 0;
#pragma unroll
            for (int b = 0; b < 8; ++b) {
                w[b] = 0;
                if (j0 + b < nb) need |= 1u << b;
            }
            const uint64_t t0 = ptx::globaltimer();
            const bool vec = (nb & 7) == 0 && j0 + 8 <= nb;   // 32-byte aligned run of 8 words
            for (;;) {
                const int gab = lane == 0 ? ld_relaxed_i32(a.gabort) : 0;
                if (vec) {
                    const uint4 lo = ld_relaxed_v4(trow + j0), hi = ld_relaxed_v4(trow + j0 + 4);
                    w[0] = lo.x; w[1] = lo.y; w[2] = lo.z; w[3] = lo.w;
                    w[4] = hi.x; w[5] = hi.y; w[6] = hi.z; w[7] = hi.w;
                } else {
#pragma unroll
                    for (int b = 0; b < 8; ++b)
                        if ((need >> b) & 1u) w[b] = ld_relaxed_u32(trow + j0 + b);
                }
#pragma unroll
                for (int b = 0; b < 8; ++b)
                    if ((w[b] >> 1) == a.epoch) need &= ~(1u << b);
                if (!__any_sync(0xffffffffu, need != 0)) break;
                if (!(ok = keep_polling(t0, gab, a, abort, lane))) break;
            }
            if (!ok) break;
            uint32_t bits = 0;
#pragma unroll
            for (int b = 0; b < 8; ++b)
                if (j0 + b < nb && (w[b] & 1u)) bits |= 1u << b;
            const int cnt = __popc(bits);
            int incl = cnt;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, incl, off);
                if (lane >= off) incl += v;
            }
            const int tot = __shfl_sync(0xffffffffu, incl, 31);
            int e = gprefix + incl - cnt;   // step-wide index of this lane's first open block
            // the lane's open blocks dealt round-robin: block e of the step goes to CTA e % Q of the slice
            // (one modulo per lane; the ABI's list is written after the pushes, off the convolution's path)
            uint32_t sel = 0;
            {
                int r = e % Q;
#pragma unroll
                for (int b = 0; b < 8; ++b) {
                    if (!((bits >> b) & 1u)) continue;
                    if (r == q) sel |= 1u << b;
                    if (++r == Q) r = 0;
                }
            }
            if (conv_cta) {
                // lane 0 pushes the selected blocks in block order, visiting only lanes that hold some
                for (uint32_t lanes = __ballot_sync(0xffffffffu, sel != 0); lanes; lanes &= lanes - 1) {
                    const int L = __ffs(lanes) - 1;
                    const uint32_t sL = __shfl_sync(0xffffffffu, sel, L);
                    if (lane == 0 && ok) {
                        const int jL = base + L * 8;
                        for (uint32_t m = sL; m && ok; m &= m - 1) ok = pr.push(n * nb + jL + (__ffs(m) - 1));
                    }
                }
                ok = __shfl_sync(0xffffffffu, (int)ok, 0) != 0;
            }
            if (owner) {
#pragma unroll
                for (int b = 0; b < 8; ++b)
                    if ((bits >> b) & 1u) a.list[e++] = n * nb + j0 + b;
            }
            gprefix += tot;
        }
        if (n == a.n - 1 && lane == 0 && ok && (int)blockIdx.x == n % (int)gridDim.x) {
            *a.count = gprefix;
            if (!a.force) *(volatile int*)a.hint = gprefix;
        }
    }
    if (lane == 0) pr.finish();
}

template <int KS, class C>
__global__ void __launch_bounds__(C::THREADS, 1)
step_fused_kernel(const __grid_constant__ CUtensorMap tm_xt, const __grid_constant__ CUtensorMap tm_xp,
                  const __grid_constant__ CUtensorMap tm_w, const __grid_constant__ CUtensorMap tm_z,
                  const FusedArgs a)
{
    using Gm = ws::Geom<KS, C::STAGES>;
    constexpr int NG = C::GATE_WARPS, NST = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = ptx::align_smem_1024(smem_raw);
    uint8_t* sX = smem;
    uint8_t* ring = sX + Gm::STAGE_BYTES;
    float* sZ = (float*)(ring + NG * FS_SLOT);
    ws::Bars* bars = (ws::Bars*)((uint8_t*)sZ + 2 * TC_ZBYTES);
    FusedShared* sh = (FusedShared*)((uint8_t*)bars + 256);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int slice = blockIdx.x % a.n_slices;
    const int ct = slice / a.n_chunks, chunk = slice % a.n_chunks;
    const int Q = gridDim.x / a.n_slices, q = blockIdx.x / a.n_slices;
    const bool conv_cta = (int)blockIdx.x < Q * a.n_slices;

    if (threadIdx.x == 0) {
        ws::init_barriers(bars);
        for (int s = 0; s < NG; ++s) ptx::mbar_init(ptx::smem_u32(&sh->g_full[s]), 1);
        ptx::fence_mbar_init();
    }
    if (warp == 9) {
        ptx::tmem_alloc(ptx::smem_u32(&bars->tmem_base), ws::TMEM_COLS);
        ptx::tmem_relinquish();
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = bars->tmem_base;
    volatile int* abort = &bars->abort;

    if (warp >= 10 + FS_BG_WARPS) {
        const int gw = warp - 10 - FS_BG_WARPS;
        if (a.log2g == 5) gate_pixels_role<5, NG>(a, sh, ring, gw, lane, abort);
        else if (a.log2g == 4) gate_pixels_role<4, NG>(a, sh, ring, gw, lane, abort);
        else gate_pixels_role<3, NG>(a, sh, ring, gw, lane, abort);
    } else if (warp >= 10) {
        gate_blocks_role<KS>(a, sh, abort, warp - 10, lane);
    } else {
        // convolution roles: the weight slice goes through the stage area into
        // TMEM first (named barrier 2 over the 10 convolution warps)
        if (conv_cta && warp < 4)
            ws::load_weight_slice<KS, NST>(&tm_w, sX, bars, tmem, a.ci_pad, chunk, ct, threadIdx.x, abort,
                                                 a.err);
        ptx::tc_fence_before();
        ptx::named_bar_sync(2, 320);
        ptx::tc_fence_after();
        if (warp == 8) {
            ws::Producer<KS, NST> pr;
            if (lane == 0) pr.init(sX, bars, &tm_xt, &tm_xp, abort, a.err, chunk, a.pad, a.nby, a.nbx);
            conv_producer_role<KS, NST>(a, pr, conv_cta, Q, q, abort, lane);
        } else if (warp == 9) {
            ws::mma_role<KS, NST>(sX, bars, tmem, abort, a.err);
        } else if (warp >= 4) {
            ws::residual_role<KS, NST>(sX, bars, threadIdx.x - 128, abort, a.err);
        } else {
            ws::epilogue_role(sZ, bars, tmem, &tm_z, ct, a.nby, a.nbx, threadIdx.x, abort, a.err, 2);
        }
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        __syncwarp();
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, ws::TMEM_COLS);
    }
}

template <int KS, class C>
cudaError_t launch_fused_ks(const Layer& L, const CUtensorMap& tm_xt, int prev_index, const FusedArgs& a)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(L.num_sms);
    cfg.blockDim = dim3(C::THREADS);
    cfg.dynamicSmemBytes = fused_smem_bytes<KS, C>();
    cfg.stream = L.stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, step_fused_kernel<KS, C>, tm_xt, L.tmap_xrow[prev_index], L.tmap_w, L.tmap_z,
                              a);
}

template <int KS, class C>
cudaError_t prepare_cfg(const Layer& L)
{
    static_assert(fused_smem_bytes<KS, C>() <= 227 * 1024, "shared memory");
    cudaError_t e = cudaFuncSetAttribute(step_fused_kernel<KS, C>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)fused_smem_bytes<KS, C>());
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, step_fused_kernel<KS, C>, C::THREADS,
                                                      fused_smem_bytes<KS, C>());
    if (e != cudaSuccess) return e;
    return per_sm >= 1 ? cudaSuccess : cudaErrorCooperativeLaunchTooLarge;
}

template <int KS>
cudaError_t prepare_ks(const Layer& L)
{
    cudaError_t e = prepare_cfg<KS, CfgSparse>(L);
    if (e == cudaSuccess) e = prepare_cfg<KS, CfgBusy>(L);
    return e != cudaSuccess ? e : prepare_cfg<KS, CfgForced>(L);
}

// The launch's form: forced steps one, sparse steps another after a sparse step that opened at least
// 3/8 of the blocks.  The hint is the count the last finished sparse step wrote into mapped host memory
// (a launch queued behind a running step reads the one before: it only chooses the form).
template <int KS>
cudaError_t launch_ks(const Layer& L, const CUtensorMap& tm_xt, int prev_index, const FusedArgs& a)
{
    if (a.force) return launch_fused_ks<KS, CfgForced>(L, tm_xt, prev_index, a);
    const long long nblk = (long long)a.n * a.nby * a.nbx;
    const int last_open = *(volatile const int*)L.open_hint_host;
    return 8LL * last_open >= 3LL * nblk ? launch_fused_ks<KS, CfgBusy>(L, tm_xt, prev_index, a)
                                         : launch_fused_ks<KS, CfgSparse>(L, tm_xt, prev_index, a);
}

}  // namespace

bool step_fused_supported(const Layer& L)
{
    if (!conv_ws_supported(L) || L.p.dtype != SKIPCONV_BF16 || L.p.stride != 1 || L.p.block != 8) return false;
    if (L.p.gate == SKIPCONV_GATE_GUMBEL) return false;   // the fused gate warps compute norms only
    const int pb = L.p.c_in * 2;
    // one 16-byte unit per gate lane, 8 to 32 lanes per pixel
    if (pb % 16 != 0 || pb / 16 > 32 || pb / 16 < 5) return false;
    if ((7 + L.p.k_h) * (7 + L.p.k_w) > FS_FOOT) return false;
    int coop = 0;
    if (cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, L.device) != cudaSuccess || !coop) return false;
    const int n_slices = (L.co_pad / TC_M) * (L.ci_pad / TC_CK);
    return n_slices <= L.num_sms;
}

cudaError_t step_fused_prepare(Layer& L)
{
    return L.p.k_h == 3 ? prepare_ks<3>(L) : prepare_ks<1>(L);
}

cudaError_t launch_step_fused(Layer& L, const void* x_t, int force)
{
    alignas(64) CUtensorMap tm_xt;
    if (!encode_xrow_map(&tm_xt, x_t, L)) {
        set_error("tensor map of x_t rejected");
        return cudaErrorInvalidValue;
    }
    // 1 .. 2^31 - 1; every step rewrites every tagged word with a max reduction, so the words go back
    // to 0 (no epoch) before the epoch wraps around to 1
    if (L.epoch == 0x7fffffffu) {
        cudaError_t e = cudaMemsetAsync(L.pnorm, 0, (size_t)L.p.n_streams * L.p.h * L.p.w * sizeof(uint64_t), L.stream);
        if (e == cudaSuccess)
            e = cudaMemsetAsync(L.gtag, 0, (size_t)L.p.n_streams * L.nby * L.nbx * sizeof(uint32_t), L.stream);
        if (e != cudaSuccess) return e;
    }
    L.epoch = L.epoch % 0x7fffffffu + 1u;
    const int cur = (int)(L.t & 1), nxt = cur ^ 1;
    FusedArgs a;
    a.xt = (const uint8_t*)x_t;
    a.xp = (const uint8_t*)L.xbuf[cur];
    a.xn = (uint4*)L.xbuf[nxt];
    a.chg_prev = L.chg[nxt];
    a.chg_cur = L.chg[cur];
    a.pnorm = L.pnorm;
    a.n = L.p.n_streams;
    a.P = L.p.h * L.p.w;
    a.W = L.p.w;
    a.H = L.p.h;
    a.pb = L.p.c_in * 2;
    a.units = a.pb / 16;
    int log2g = 0;
    while ((1 << log2g) < a.units) ++log2g;
    a.log2g = log2g;
    a.gch = 8 * (32 >> log2g);   // 8 rows of 32 / G pixels
    a.mask = L.mask;
    a.gtag = L.gtag;
    a.list = L.list;
    a.count = step_count(L);
    a.hint = L.open_hint_dev;
    a.gabort = L.sched;
    a.epoch = L.epoch;
    a.thr = L.gate_thr;
    a.force = force;
    a.Ho = L.ho;
    a.Wo = L.wo;
    a.KH = L.p.k_h;
    a.KW = L.p.k_w;
    a.pad = L.p.pad;
    a.nby = L.nby;
    a.nbx = L.nbx;
    a.err = L.err_dev;
    a.ci_pad = L.ci_pad;
    a.n_chunks = L.ci_pad / TC_CK;
    a.n_slices = (L.co_pad / TC_M) * a.n_chunks;
    return L.p.k_h == 3 ? launch_ks<3>(L, tm_xt, cur, a) : launch_ks<1>(L, tm_xt, cur, a);
}

}  // namespace sc
