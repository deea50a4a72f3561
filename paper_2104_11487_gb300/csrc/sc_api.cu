// Host side of the Skip-Conv C ABI (include/skipconv.h): argument checks,
// state allocation, weight repacking, and the per-step launch sequence
//   step_fused (one cooperative tensor-core launch), or
//   step_local (one CUDA-core launch, a CTA per tile of gate blocks), or
//   gate_pixel -> gate_block -> conv (tensor-core or CUDA-core) [-> y_refresh]
// all on the handle's stream, with no host synchronisation per step.
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <mutex>
#include <new>
#include <vector>

#include "sc_internal.h"
#include "sc_ptx.cuh"

namespace sc {

int gate_max_channels(int dtype, bool vec);

static thread_local char g_last_error[512];

void set_error(const char* fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
    va_end(ap);
}

// cudaFuncAttributeMaxDynamicSharedMemorySize belongs to the kernel, not to a
// layer: layers that share a kernel but need different amounts must only ever
// raise it, or the last layer created would lower it below what an earlier
// one launches with.
cudaError_t ensure_dynamic_smem(const void* func, size_t bytes)
{
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, func);
    if (e != cudaSuccess) return e;
    if ((size_t)fa.maxDynamicSharedSizeBytes >= bytes) return cudaSuccess;
    return cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

EncodeTiledFn encode_tiled_fn()
{
    static EncodeTiledFn fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)p;
    }
    return fn;
}

// Host-side fault injection for the cleanup paths: SKIPCONV_FAULT_ALLOC=k
// makes the k-th device allocation of skipconv_create fail (k >= 1).
static int fault_alloc_index()
{
    const char* s = getenv("SKIPCONV_FAULT_ALLOC");
    return s ? atoi(s) : 0;
}

struct Allocator {
    int counter = 0;
    int fail_at = 0;
    size_t bytes = 0;
    cudaError_t dev(void** p, size_t n)
    {
        ++counter;
        if (fail_at > 0 && counter == fail_at) {
            *p = nullptr;
            return cudaErrorMemoryAllocation;
        }
        cudaError_t e = cudaMalloc(p, n < 16 ? 16 : n);
        if (e == cudaSuccess) bytes += n;
        return e;
    }
};

static void prof_release(Layer* L)
{
    if (L->prof_ev) {
        for (int i = 0; i < 2 * L->prof_cap; ++i)
            if (L->prof_ev[i]) cudaEventDestroy(L->prof_ev[i]);
        free(L->prof_ev);
    }
    free(L->prof_kind);
    L->prof_ev = nullptr;
    L->prof_kind = nullptr;
    L->prof_cap = L->prof_n = 0;
}

// Record the event opening a timed launch of `kind`; returns the slot or -1.
static int prof_begin(Layer* L, int kind)
{
    L->launches[kind] += 1;
    if (!L->prof_on) return -1;
    if (L->prof_n == L->prof_cap) {
        const int cap = L->prof_cap ? 2 * L->prof_cap : 256;
        cudaEvent_t* ev = (cudaEvent_t*)calloc(2 * (size_t)cap, sizeof(cudaEvent_t));
        int* kinds = (int*)calloc(cap, sizeof(int));
        if (!ev || !kinds) {
            free(ev);
            free(kinds);
            return -1;
        }
        if (L->prof_ev) memcpy(ev, L->prof_ev, 2 * (size_t)L->prof_cap * sizeof(cudaEvent_t));
        if (L->prof_kind) memcpy(kinds, L->prof_kind, (size_t)L->prof_cap * sizeof(int));
        free(L->prof_ev);
        free(L->prof_kind);
        L->prof_ev = ev;
        L->prof_kind = kinds;
        L->prof_cap = cap;
    }
    const int i = L->prof_n;
    for (int k = 0; k < 2; ++k)
        if (!L->prof_ev[2 * i + k] && cudaEventCreate(&L->prof_ev[2 * i + k]) != cudaSuccess) return -1;
    L->prof_kind[i] = kind;
    if (cudaEventRecord(L->prof_ev[2 * i], L->stream) != cudaSuccess) return -1;
    return i;
}

static void prof_end(Layer* L, int slot)
{
    if (slot < 0) return;
    if (cudaEventRecord(L->prof_ev[2 * slot + 1], L->stream) == cudaSuccess) L->prof_n = slot + 1;
}

static void free_buffers(Layer* L)
{
    prof_release(L);
    void* ptrs[] = {L->xbuf[0], L->xbuf[1], L->chg[0], L->chg[1], L->pix_l1, L->mask, L->list, L->counters,
                    L->z, L->y, L->bias, L->w_cc, L->w_tc, L->x_stage, L->sched, L->pnorm, L->gtag,
                    L->pix_taps, L->gphi, L->w_loc, L->ychg, L->tile_chg, L->z_prev, L->tx};
    for (void* p : ptrs)
        if (p) cudaFree(p);
    if (L->err_host) cudaFreeHost(L->err_host);
}

static int status_of(cudaError_t e)
{
    if (e == cudaSuccess) return SKIPCONV_OK;
    cudaGetLastError();  // clear a sticky launch error so the next call starts clean
    set_error("CUDA error %d: %s", (int)e, cudaGetErrorString(e));
    return e == cudaErrorMemoryAllocation ? SKIPCONV_ERR_OOM : SKIPCONV_ERR_CUDA;
}

static int check_device_word(const Layer* L)
{
    const int v = *(volatile int*)L->err_host;
    if (v == DEV_OK) return SKIPCONV_OK;
    set_error("device error word %d", v);
    return v == DEV_TIMEOUT ? SKIPCONV_ERR_TIMEOUT : SKIPCONV_ERR_DEVICE;
}

int validate(const skipconv_params* p)
{
    if (!p) return set_error("params is NULL"), SKIPCONV_ERR_INVALID;
    if (p->n_streams < 1 || p->c_in < 1 || p->c_out < 1 || p->h < 1 || p->w < 1 || p->k_h < 1 || p->k_w < 1 ||
        p->stride < 1 || p->pad < 0 || p->groups < 1 || p->block < 1)
        return set_error("non-positive size in params"), SKIPCONV_ERR_INVALID;
    if (p->c_in % p->groups || p->c_out % p->groups)
        return set_error("c_in and c_out must be divisible by groups"), SKIPCONV_ERR_INVALID;
    if (p->h + 2 * p->pad < p->k_h || p->w + 2 * p->pad < p->k_w)
        return set_error("kernel larger than the padded frame"), SKIPCONV_ERR_INVALID;
    if (!(p->eps >= 0.f)) return set_error("eps must be >= 0"), SKIPCONV_ERR_INVALID;
    if (p->key_interval < 0) return set_error("key_interval must be >= 0"), SKIPCONV_ERR_INVALID;
    if (p->gate < SKIPCONV_GATE_INPUT_MEAN || p->gate > SKIPCONV_GATE_GUMBEL)
        return set_error("unknown gate %d", p->gate), SKIPCONV_ERR_INVALID;
    if (p->dtype != SKIPCONV_F32 && p->dtype != SKIPCONV_BF16)
        return set_error("unknown dtype %d", p->dtype), SKIPCONV_ERR_INVALID;
    if (p->activation < SKIPCONV_ACT_NONE || p->activation > SKIPCONV_ACT_SILU)
        return set_error("unknown activation %d", p->activation), SKIPCONV_ERR_INVALID;
    if (p->conv_path < SKIPCONV_PATH_AUTO || p->conv_path > SKIPCONV_PATH_CUDA_CORE_SEPARATE)
        return set_error("unknown conv_path %d", p->conv_path), SKIPCONV_ERR_INVALID;
    const long long frame = (long long)p->n_streams * p->h * p->w;
    if (frame * p->c_in > (1LL << 40)) return set_error("frame too large"), SKIPCONV_ERR_INVALID;
    const int ho = (p->h + 2 * p->pad - p->k_h) / p->stride + 1;
    const int wo = (p->w + 2 * p->pad - p->k_w) / p->stride + 1;
    const long long nblocks = (long long)p->n_streams * ((ho + p->block - 1) / p->block) * ((wo + p->block - 1) / p->block);
    if (nblocks >= (1LL << 31)) return set_error("too many gate blocks"), SKIPCONV_ERR_INVALID;
    if (p->gate == SKIPCONV_GATE_GUMBEL &&
        (p->k_h * p->k_w > 9 || (size_t)p->k_h * p->k_w * p->c_in * sizeof(float) > 48 * 1024))
        return set_error("Gumbel gate: at most 9 taps and taps*c_in*4 <= 48 KiB"), SKIPCONV_ERR_UNSUPPORTED;
    if (p->c_in > gate_max_channels(p->dtype, false))
        return set_error("c_in above %d", gate_max_channels(p->dtype, false)), SKIPCONV_ERR_UNSUPPORTED;
    return SKIPCONV_OK;
}

}  // namespace sc

using namespace sc;

struct skipconv_s {
    Layer L;
};

static Layer* get(skipconv_handle h) { return h ? &h->L : nullptr; }

// Live layers, so that destroying a layer can drop the links other layers hold to it.
static std::mutex& live_mu()
{
    static std::mutex mu;
    return mu;
}
static std::vector<Layer*>& live_layers()
{
    static std::vector<Layer*> v;
    return v;
}

extern "C" {

const char* skipconv_status_string(int s)
{
    switch (s) {
    case SKIPCONV_OK: return "SKIPCONV_OK";
    case SKIPCONV_ERR_INVALID: return "SKIPCONV_ERR_INVALID";
    case SKIPCONV_ERR_UNSUPPORTED: return "SKIPCONV_ERR_UNSUPPORTED";
    case SKIPCONV_ERR_CUDA: return "SKIPCONV_ERR_CUDA";
    case SKIPCONV_ERR_OOM: return "SKIPCONV_ERR_OOM";
    case SKIPCONV_ERR_TIMEOUT: return "SKIPCONV_ERR_TIMEOUT";
    case SKIPCONV_ERR_DEVICE: return "SKIPCONV_ERR_DEVICE";
    default: return "SKIPCONV_UNKNOWN_STATUS";
    }
}

const char* skipconv_last_error(void) { return g_last_error; }

int skipconv_create(const skipconv_params* params, const void* weights_oihw, const float* bias, void* stream,
                    skipconv_handle* out)
{
    if (!out) return set_error("out is NULL"), SKIPCONV_ERR_INVALID;
    *out = nullptr;
    int st = validate(params);
    if (st) return st;
    if (!weights_oihw) return set_error("weights is NULL"), SKIPCONV_ERR_INVALID;

    skipconv_s* h = new (std::nothrow) skipconv_s();
    if (!h) return set_error("host allocation failed"), SKIPCONV_ERR_OOM;
    Layer& L = h->L;
    memset(&L, 0, sizeof(L));
    L.p = *params;
    L.stream = (cudaStream_t)stream;
    L.ho = (L.p.h + 2 * L.p.pad - L.p.k_h) / L.p.stride + 1;
    L.wo = (L.p.w + 2 * L.p.pad - L.p.k_w) / L.p.stride + 1;
    L.nby = (L.ho + L.p.block - 1) / L.p.block;
    L.nbx = (L.wo + L.p.block - 1) / L.p.block;
    L.cpg = L.p.c_in / L.p.groups;
    L.opg = L.p.c_out / L.p.groups;
    L.esize = L.p.dtype == SKIPCONV_BF16 ? 2 : 4;

    cudaError_t e = cudaGetDevice(&L.device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&L.num_sms, cudaDevAttrMultiProcessorCount, L.device);
    if (e != cudaSuccess) {
        st = status_of(e);
        delete h;
        return st;
    }

    // choose the convolution path
    const char* why = "";
    const bool tc_ok = conv_tc_supported(L.p, &why);
    const bool want_tc = L.p.conv_path == SKIPCONV_PATH_TENSOR_CORE ||
                         L.p.conv_path == SKIPCONV_PATH_TENSOR_CORE_SEPARATE;
    if (want_tc && !tc_ok) {
        set_error("tensor-core path unsupported: %s", why);
        delete h;
        return SKIPCONV_ERR_UNSUPPORTED;
    }
    const bool want_cc = L.p.conv_path == SKIPCONV_PATH_CUDA_CORE ||
                         L.p.conv_path == SKIPCONV_PATH_CUDA_CORE_SEPARATE;
    // AUTO: small layers (latency-bound steps) take the one-launch step, a CTA per tile of gate
    // blocks; its contraction runs on the tensor cores for dense bf16 layers (depthwise and fp32
    // layers keep the CUDA cores)
    const bool small = L.p.conv_path == SKIPCONV_PATH_AUTO && step_local_preferred(L);
    L.path = (want_cc || small || !tc_ok) ? SKIPCONV_PATH_CUDA_CORE : SKIPCONV_PATH_TENSOR_CORE;
    L.local_tc = (L.p.conv_path == SKIPCONV_PATH_AUTO && L.path == SKIPCONV_PATH_CUDA_CORE &&
                  L.p.dtype == SKIPCONV_BF16 && L.p.groups == 1 && !(L.cpg == 1 && L.opg == 1))
                     ? 1
                     : 0;
    L.ci_pad = ((L.p.c_in + 63) / 64) * 64;
    L.co_pad = ((L.p.c_out + 127) / 128) * 128;

    Allocator A;
    A.fail_at = fault_alloc_index();
    const size_t npix = (size_t)L.p.n_streams * L.p.h * L.p.w;
    const size_t xbytes = npix * L.p.c_in * L.esize;
    const size_t nz = (size_t)L.p.n_streams * L.ho * L.wo * L.p.c_out;
    const size_t nblk = (size_t)L.p.n_streams * L.nby * L.nbx;
    const size_t nw = (size_t)L.p.c_out * L.cpg * L.p.k_h * L.p.k_w;
    double* w_l1_dev = nullptr;
    e = cudaSuccess;
    if (e == cudaSuccess) e = A.dev(&L.xbuf[0], xbytes);
    if (e == cudaSuccess) e = A.dev(&L.xbuf[1], xbytes);
    if (e == cudaSuccess) e = A.dev((void**)&L.chg[0], npix);
    if (e == cudaSuccess) e = A.dev((void**)&L.chg[1], npix);
    if (e == cudaSuccess) e = A.dev((void**)&L.pix_l1, npix * sizeof(float));
    if (e == cudaSuccess && L.p.gate == SKIPCONV_GATE_GUMBEL) {
        const size_t taps = (size_t)L.p.k_h * L.p.k_w;
        e = A.dev((void**)&L.pix_taps, npix * taps * sizeof(float));
        if (e == cudaSuccess) e = A.dev((void**)&L.gphi, taps * L.p.c_in * sizeof(float));
        if (e == cudaSuccess) e = gumbel_prepare(L);
    }
    if (e == cudaSuccess) e = A.dev((void**)&L.mask, nblk);
    if (e == cudaSuccess) e = A.dev((void**)&L.list, nblk * sizeof(int32_t));
    if (e == cudaSuccess) e = A.dev((void**)&L.counters, 64 * sizeof(int32_t));
    if (e == cudaSuccess) e = A.dev((void**)&L.z, nz * sizeof(float));
    if (e == cudaSuccess && L.p.emit_y) e = A.dev(&L.y, nz * L.esize);
    if (e == cudaSuccess) e = A.dev((void**)&L.bias, L.p.c_out * sizeof(float));
    if (e == cudaSuccess) e = A.dev((void**)&L.w_cc, nw * sizeof(float));
    if (e == cudaSuccess && L.path == SKIPCONV_PATH_TENSOR_CORE)
        e = A.dev((void**)&L.w_tc, (size_t)L.co_pad * L.p.k_h * L.p.k_w * L.ci_pad * sizeof(__nv_bfloat16));
    if (e == cudaSuccess) e = A.dev((void**)&w_l1_dev, sizeof(double));
    if (e == cudaSuccess) {
        // the device error word and, a cache line further, the fused step's open-block hint
        e = cudaHostAlloc((void**)&L.err_host, 32 * sizeof(int), cudaHostAllocMapped);
        if (e == cudaSuccess) {
            memset(L.err_host, 0, 32 * sizeof(int));
            e = cudaHostGetDevicePointer((void**)&L.err_dev, L.err_host, 0);
            L.open_hint_host = L.err_host + 16;
            L.open_hint_dev = L.err_dev + 16;
        }
    }
    L.state_bytes = A.bytes;
    if (e != cudaSuccess) {
        st = status_of(e);
        if (w_l1_dev) cudaFree(w_l1_dev);
        free_buffers(&h->L);
        delete h;
        return st;
    }

    // weights, bias, ||w||_1
    double w_l1 = 0.0;
    e = cudaMemsetAsync(w_l1_dev, 0, sizeof(double), L.stream);
    if (e == cudaSuccess && L.w_tc)
        e = cudaMemsetAsync(L.w_tc, 0, (size_t)L.co_pad * L.p.k_h * L.p.k_w * L.ci_pad * sizeof(__nv_bfloat16),
                            L.stream);
    if (e == cudaSuccess) e = launch_pack_weights(L, weights_oihw, w_l1_dev);
    if (e == cudaSuccess) {
        if (bias)
            e = cudaMemcpyAsync(L.bias, bias, L.p.c_out * sizeof(float), cudaMemcpyDeviceToDevice, L.stream);
        else
            e = cudaMemsetAsync(L.bias, 0, L.p.c_out * sizeof(float), L.stream);
    }
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(&w_l1, w_l1_dev, sizeof(double), cudaMemcpyDeviceToHost, L.stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(L.stream);
    cudaFree(w_l1_dev);
    (void)nw;

    // The gate compares the raw local l1 sum S (sum of |r| over the support) with
    // a threshold equivalent to the chosen normalisation of Eq. 5 / Eq. 7.
    double thr;
    if (L.p.gate == SKIPCONV_GATE_INPUT_MEAN) thr = (double)L.p.eps * L.p.c_in * L.p.k_h * L.p.k_w;
    else if (L.p.gate == SKIPCONV_GATE_INPUT_SUM) thr = (double)L.p.eps;
    else if (L.p.gate == SKIPCONV_GATE_GUMBEL) thr = (double)L.p.eps;
    else thr = w_l1 > 0.0 ? (double)L.p.eps / w_l1 : INFINITY;
    L.gate_thr = (float)thr;

    if (e == cudaSuccess && L.path == SKIPCONV_PATH_TENSOR_CORE) e = conv_tc_prepare(L);
    if (e == cudaSuccess && L.path == SKIPCONV_PATH_TENSOR_CORE && conv_ws_supported(L)) {
        e = conv_ws_prepare(L);
        L.tc_ws = e == cudaSuccess ? 1 : 0;
    }
    // the whole step as one cooperative launch, unless the separate launches were asked for
    if (e == cudaSuccess && L.tc_ws && L.p.conv_path != SKIPCONV_PATH_TENSOR_CORE_SEPARATE &&
        step_fused_supported(L)) {
        e = A.dev((void**)&L.sched, 16 * sizeof(int));
        if (e == cudaSuccess) e = A.dev((void**)&L.pnorm, npix * sizeof(uint64_t));
        if (e == cudaSuccess) e = A.dev((void**)&L.gtag, nblk * sizeof(uint32_t));
        // tags start at 0, which no step uses
        if (e == cudaSuccess) e = cudaMemsetAsync(L.pnorm, 0, npix * sizeof(uint64_t), L.stream);
        if (e == cudaSuccess) e = cudaMemsetAsync(L.gtag, 0, nblk * sizeof(uint32_t), L.stream);
        if (e == cudaSuccess) {
            const cudaError_t pe = step_fused_prepare(L);
            if (pe == cudaSuccess) {
                L.fused = 1;
            } else {
                cudaGetLastError();   // not fatal: the separate launches serve this layer
            }
        }
        L.state_bytes = A.bytes;
    }
    // CUDA-core layers: the whole step as one launch, unless the separate launches were asked for
    if (e == cudaSuccess && step_local_supported(L)) {
        e = step_local_prepare(L);
        if (e == cudaSuccess) L.fused = 2;
    }
    if (e == cudaSuccess) {
        h->L.key = 1;
        st = skipconv_reset_state(h);
        if (st == SKIPCONV_OK) e = cudaStreamSynchronize(L.stream);
        else e = cudaErrorUnknown;
    }
    if (e != cudaSuccess) {
        st = st ? st : status_of(e);
        free_buffers(&h->L);
        delete h;
        return st;
    }
    {
        std::lock_guard<std::mutex> lock(live_mu());
        live_layers().push_back(&h->L);
    }
    *out = h;
    return SKIPCONV_OK;
}

int skipconv_reset_state(skipconv_handle h)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    if (int st = check_device_word(L)) return st;
    const size_t npix = (size_t)L->p.n_streams * L->p.h * L->p.w;
    const size_t xbytes = npix * L->p.c_in * L->esize;
    cudaError_t e = cudaMemsetAsync(L->xbuf[0], 0, xbytes, L->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(L->xbuf[1], 0, xbytes, L->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(L->chg[0], 0, npix, L->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(L->chg[1], 0, npix, L->stream);
    if (e == cudaSuccess) e = cudaMemsetAsync(L->counters, 0, 64 * sizeof(int32_t), L->stream);
    if (e == cudaSuccess && L->sched) e = cudaMemsetAsync(L->sched, 0, 16 * sizeof(int), L->stream);
    if (e == cudaSuccess) e = launch_reset_z(*L);
    if (e == cudaSuccess && L->y) e = cudaMemsetAsync(L->y, 0, (size_t)L->p.n_streams * L->ho * L->wo * L->p.c_out * L->esize, L->stream);
    if (e == cudaSuccess && L->tile_chg) e = cudaMemsetAsync(L->tile_chg, 0, 2 * (size_t)L->ntiles, L->stream);
    if (e != cudaSuccess) return status_of(e);
    L->t = 0;
    L->key = 1;
    return SKIPCONV_OK;
}

int skipconv_step(skipconv_handle h, const void* x_t, const void* shortcut)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    if (!x_t) return set_error("x_t is NULL"), SKIPCONV_ERR_INVALID;
    if ((uintptr_t)x_t % 16 || (uintptr_t)shortcut % 16)
        return set_error("x_t and shortcut must be 16-byte aligned"), SKIPCONV_ERR_INVALID;
    if (shortcut && !L->y) return set_error("shortcut given but the layer keeps no y (emit_y = 0)"), SKIPCONV_ERR_INVALID;
    if (int st = check_device_word(L)) return st;
    if (L->p.gate == SKIPCONV_GATE_GUMBEL && !L->gphi_set)
        return set_error("Gumbel gate: call skipconv_set_gate_weights before the first step"), SKIPCONV_ERR_INVALID;
    if (L->p.key_interval > 0 && !L->key && L->since_key >= L->p.key_interval) {
        const int st = skipconv_reset_state(h);   // periodic key frame (Table 4)
        if (st != SKIPCONV_OK) return st;
    }
    const int cur = (int)(L->t & 1), nxt = cur ^ 1;
    // xbuf[cur] holds x_{t-1}; xbuf[nxt] holds x_{t-2} and receives x_t.
    // chg[nxt] marks pixels that changed at the previous step; chg[cur] is written now.
    const int force = (L->key || L->p.dense_mode) ? 1 : 0;
    if (L->fused) {
        const int kind = L->fused == 1 ? 4 : 5;
        // stack propagation: a linked producer's change flags describe this x_t (or shortcut) only
        // when it is that producer's y and the producer stepped exactly once since this layer did
        const Layer* px = (L->link_x && x_t == L->link_x->y && L->link_x->steps == L->link_x_seen + 1) ? L->link_x
                                                                                                      : nullptr;
        const Layer* psc = (shortcut && L->link_sc && shortcut == L->link_sc->y &&
                            L->link_sc->steps == L->link_sc_seen + 1)
                               ? L->link_sc
                               : nullptr;
        const int slot = prof_begin(L, kind);
        const cudaError_t e = L->fused == 1 ? launch_step_fused(*L, x_t, force)
                                            : launch_step_local(*L, x_t, shortcut, force, px, psc);
        prof_end(L, slot);
        if (e != cudaSuccess) return status_of(e);
        L->since_key = force && L->key ? 1 : L->since_key + 1;
        L->t += 1;
        L->key = 0;
        L->steps += 1;
        if (L->link_x) L->link_x_seen = L->link_x->steps;
        if (L->link_sc) L->link_sc_seen = L->link_sc->steps;
        return SKIPCONV_OK;
    }
    const bool gumbel = L->p.gate == SKIPCONV_GATE_GUMBEL;
    int slot = prof_begin(L, 0);
    cudaError_t e = gumbel ? launch_gate_pixels_gumbel(*L, x_t, L->xbuf[cur], L->xbuf[nxt], L->chg[nxt], L->chg[cur])
                           : launch_gate_pixels(*L, x_t, L->xbuf[cur], L->xbuf[nxt], L->chg[nxt], L->chg[cur], force);
    prof_end(L, slot);
    if (e == cudaSuccess) {
        slot = prof_begin(L, 1);
        e = gumbel ? launch_gate_blocks_gumbel(*L, force) : launch_gate_blocks(*L, force);
        prof_end(L, slot);
    }
    if (e == cudaSuccess) {
        slot = prof_begin(L, 2);
        if (L->path == SKIPCONV_PATH_TENSOR_CORE && L->tc_ws) e = launch_conv_ws(*L, x_t, cur);
        else if (L->path == SKIPCONV_PATH_TENSOR_CORE) e = launch_conv_tc(*L, x_t, L->xbuf[cur], cur);
        else e = launch_conv_cc(*L, x_t, L->xbuf[cur]);
        prof_end(L, slot);
    }
    if (e == cudaSuccess && L->y && shortcut) {
        slot = prof_begin(L, 3);
        e = launch_y_refresh(*L, shortcut);
        prof_end(L, slot);
    }
    if (e != cudaSuccess) return status_of(e);
    L->since_key = force && L->key ? 1 : L->since_key + 1;
    L->t += 1;
    L->key = 0;
    L->steps += 1;
    return SKIPCONV_OK;
}

int skipconv_step_warped(skipconv_handle h, const void* x_t, const void* shortcut, const float* flow)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    if (!x_t || !flow) return set_error("x_t and flow must not be NULL"), SKIPCONV_ERR_INVALID;
    if ((uintptr_t)x_t % 16 || (uintptr_t)shortcut % 16 || (uintptr_t)flow % 4)
        return set_error("x_t and shortcut must be 16-byte aligned, flow 4-byte aligned"), SKIPCONV_ERR_INVALID;
    if (shortcut && !L->y) return set_error("shortcut given but the layer keeps no y (emit_y = 0)"), SKIPCONV_ERR_INVALID;
    if (!step_local_warp_supported(*L))
        return set_error("warped residuals need a layer on the one-launch CUDA-core step that keeps the frame "
                         "size (stride 1, ho = h, wo = w)"),
               SKIPCONV_ERR_UNSUPPORTED;
    if (int st = check_device_word(L)) return st;
    if (L->p.key_interval > 0 && !L->key && L->since_key >= L->p.key_interval) {
        const int st = skipconv_reset_state(h);   // periodic key frame (Table 4)
        if (st != SKIPCONV_OK) return st;
    }
    // a key frame has no previous frame to warp: it is the plain key-frame step
    if (L->key) return skipconv_step(h, x_t, shortcut);
    const int cur = (int)(L->t & 1);
    // z~_t = T~(z~_{t-1}) everywhere, then + w * r_t at the open blocks with r_t = x_t - T(x_{t-1})
    int slot = prof_begin(L, 6);
    cudaError_t e = launch_step_warp_pass(*L, x_t, shortcut, flow);
    prof_end(L, slot);
    if (e == cudaSuccess) {
        slot = prof_begin(L, 5);
        e = launch_step_local(*L, x_t, shortcut, L->p.dense_mode ? 1 : 0, nullptr, nullptr, flow);
        prof_end(L, slot);
    }
    // y moved everywhere, and this form keeps no per-tile commit flags: tell linked layers (and this
    // layer's next linked step) to read whole frames
    if (e == cudaSuccess && L->ychg)
        e = cudaMemsetAsync(L->ychg, 1, (size_t)L->p.n_streams * L->nby * L->nbx, L->stream);
    if (e == cudaSuccess && L->tile_chg) e = cudaMemsetAsync(L->tile_chg + (size_t)cur * L->ntiles, 1, L->ntiles, L->stream);
    if (e != cudaSuccess) return status_of(e);
    L->since_key += 1;
    L->t += 1;
    L->steps += 1;
    if (L->link_x) L->link_x_seen = L->link_x->steps;
    if (L->link_sc) L->link_sc_seen = L->link_sc->steps;
    return SKIPCONV_OK;
}

int skipconv_link_inputs(skipconv_handle h, skipconv_handle producer_x, skipconv_handle producer_sc)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    Layer* px = get(producer_x);
    Layer* psc = get(producer_sc);
    if (px == L || psc == L) return set_error("a layer cannot be linked to itself"), SKIPCONV_ERR_INVALID;
    if (!px && psc) return set_error("a shortcut link needs the x_t link"), SKIPCONV_ERR_INVALID;
    if (px) {
        if (L->fused != 2 || !L->local_staged)
            return set_error("stack propagation needs this layer on the one-launch CUDA-core step"),
                   SKIPCONV_ERR_UNSUPPORTED;
        for (const Layer* P : {px, psc}) {
            if (!P) continue;
            if (P->fused != 2 || !P->ychg)
                return set_error("a linked producer must keep y and run the one-launch CUDA-core step"),
                       SKIPCONV_ERR_UNSUPPORTED;
            if (P->stream != L->stream) return set_error("linked layers must share the stream"), SKIPCONV_ERR_INVALID;
            if (P->p.n_streams != L->p.n_streams || P->p.dtype != L->p.dtype)
                return set_error("linked layers differ in streams or dtype"), SKIPCONV_ERR_INVALID;
        }
        if (px->ho != L->p.h || px->wo != L->p.w || px->p.c_out != L->p.c_in)
            return set_error("x_t producer's y is [n][%d][%d][%d], this layer's x_t [n][%d][%d][%d]", px->ho, px->wo,
                             px->p.c_out, L->p.h, L->p.w, L->p.c_in),
                   SKIPCONV_ERR_INVALID;
        if (psc && (psc->ho != L->ho || psc->wo != L->wo || psc->p.c_out != L->p.c_out))
            return set_error("shortcut producer's y is [n][%d][%d][%d], this layer's output [n][%d][%d][%d]", psc->ho,
                             psc->wo, psc->p.c_out, L->ho, L->wo, L->p.c_out),
                   SKIPCONV_ERR_INVALID;
    }
    std::lock_guard<std::mutex> lock(live_mu());
    L->link_x = px;
    L->link_sc = psc;
    // the first step that may use a link is the one after the producer's next step
    L->link_x_seen = px ? px->steps : 0;
    L->link_sc_seen = psc ? psc->steps : 0;
    return SKIPCONV_OK;
}

int skipconv_set_gate_weights(skipconv_handle h, const float* phi_oihw, float phi_bias)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    if (!phi_oihw) return set_error("phi is NULL"), SKIPCONV_ERR_INVALID;
    if (L->p.gate != SKIPCONV_GATE_GUMBEL)
        return set_error("skipconv_set_gate_weights: the layer's gate is not SKIPCONV_GATE_GUMBEL"),
               SKIPCONV_ERR_INVALID;
    const int taps = L->p.k_h * L->p.k_w, C = L->p.c_in;
    std::vector<float> src((size_t)taps * C), dst((size_t)taps * C);
    cudaError_t e = cudaStreamSynchronize(L->stream);
    if (e == cudaSuccess) e = cudaMemcpy(src.data(), phi_oihw, src.size() * sizeof(float), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return status_of(e);
    for (int c = 0; c < C; ++c)            // [c][kh][kw] -> [tap][c]
        for (int t = 0; t < taps; ++t) dst[(size_t)t * C + c] = src[(size_t)c * taps + t];
    e = cudaMemcpy(L->gphi, dst.data(), dst.size() * sizeof(float), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return status_of(e);
    L->gphi_bias = phi_bias;
    L->gphi_set = 1;
    return SKIPCONV_OK;
}

int skipconv_step_host(skipconv_handle h, const void* x_t_host, float* z_out_host)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    if (!x_t_host) return set_error("x_t_host is NULL"), SKIPCONV_ERR_INVALID;
    const size_t xbytes = (size_t)L->p.n_streams * L->p.h * L->p.w * L->p.c_in * L->esize;
    cudaError_t e = cudaSuccess;
    if (!L->x_stage) {
        e = cudaMalloc(&L->x_stage, xbytes);
        if (e != cudaSuccess) {
            L->x_stage = nullptr;
            return status_of(e);
        }
        L->state_bytes += xbytes;
    }
    e = cudaMemcpyAsync(L->x_stage, x_t_host, xbytes, cudaMemcpyHostToDevice, L->stream);
    if (e != cudaSuccess) return status_of(e);
    int st = skipconv_step(h, L->x_stage, nullptr);
    if (st) return st;
    if (z_out_host) {
        const size_t zbytes = (size_t)L->p.n_streams * L->ho * L->wo * L->p.c_out * sizeof(float);
        e = cudaMemcpyAsync(z_out_host, L->z, zbytes, cudaMemcpyDeviceToHost, L->stream);
        if (e != cudaSuccess) return status_of(e);
    }
    e = cudaStreamSynchronize(L->stream);
    if (e != cudaSuccess) return status_of(e);
    return check_device_word(L);
}

static void async_release(Layer* L);

// Copy streams, events and staging buffers of the pipelined host step (first call).
static cudaError_t async_prepare(Layer* L)
{
    if (L->up_stream) return cudaSuccess;
    const size_t xbytes = (size_t)L->p.n_streams * L->p.h * L->p.w * L->p.c_in * L->esize;
    const size_t zbytes = (size_t)L->p.n_streams * L->ho * L->wo * L->p.c_out * sizeof(float);
    cudaError_t e = cudaSuccess;
    for (int s = 0; s < 2 && e == cudaSuccess; ++s) {
        e = cudaMalloc(&L->xs_async[s], xbytes);
        if (e != cudaSuccess) L->xs_async[s] = nullptr;
        if (e == cudaSuccess) {
            e = cudaMalloc((void**)&L->zs_async[s], zbytes);
            if (e != cudaSuccess) L->zs_async[s] = nullptr;
        }
        for (cudaEvent_t* ev : {&L->ev_up[s], &L->ev_used[s], &L->ev_zready[s], &L->ev_down[s]})
            if (e == cudaSuccess) e = cudaEventCreateWithFlags(ev, cudaEventDisableTiming);
    }
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&L->down_stream, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&L->up_stream, cudaStreamNonBlocking);
    if (e == cudaSuccess) L->state_bytes += 2 * (xbytes + zbytes);
    else async_release(L);
    return e;
}

static void async_release(Layer* L)
{
    for (cudaStream_t st : {L->up_stream, L->down_stream})
        if (st) {
            cudaStreamSynchronize(st);
            cudaStreamDestroy(st);
        }
    L->up_stream = L->down_stream = nullptr;
    for (int s = 0; s < 2; ++s) {
        for (cudaEvent_t ev : {L->ev_up[s], L->ev_used[s], L->ev_zready[s], L->ev_down[s]})
            if (ev) cudaEventDestroy(ev);
        L->ev_up[s] = L->ev_used[s] = L->ev_zready[s] = L->ev_down[s] = nullptr;
        if (L->xs_async[s]) cudaFree(L->xs_async[s]);
        if (L->zs_async[s]) cudaFree(L->zs_async[s]);
        L->xs_async[s] = nullptr;
        L->zs_async[s] = nullptr;
    }
}

int skipconv_step_host_async(skipconv_handle h, const void* x_t_host, float* z_out_host)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    if (!x_t_host) return set_error("x_t_host is NULL"), SKIPCONV_ERR_INVALID;
    cudaError_t e = async_prepare(L);
    if (e != cudaSuccess) return status_of(e);
    const size_t xbytes = (size_t)L->p.n_streams * L->p.h * L->p.w * L->p.c_in * L->esize;
    const size_t zbytes = (size_t)L->p.n_streams * L->ho * L->wo * L->p.c_out * sizeof(float);
    const int s = (int)(L->async_steps & 1);
    // upload into staging frame s once the step two calls back has read it (an event never recorded
    // is complete, so the first two calls do not wait)
    e = cudaStreamWaitEvent(L->up_stream, L->ev_used[s], 0);
    if (e == cudaSuccess) e = cudaMemcpyAsync(L->xs_async[s], x_t_host, xbytes, cudaMemcpyHostToDevice, L->up_stream);
    if (e == cudaSuccess) e = cudaEventRecord(L->ev_up[s], L->up_stream);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(L->stream, L->ev_up[s], 0);
    if (e != cudaSuccess) return status_of(e);
    int st = skipconv_step(h, L->xs_async[s], nullptr);
    if (st) return st;
    e = cudaEventRecord(L->ev_used[s], L->stream);
    if (e == cudaSuccess && z_out_host) {
        // z after this step into staging buffer s (free once the download two calls back is done),
        // then to the host on the download stream
        e = cudaStreamWaitEvent(L->stream, L->ev_down[s], 0);
        if (e == cudaSuccess) e = cudaMemcpyAsync(L->zs_async[s], L->z, zbytes, cudaMemcpyDeviceToDevice, L->stream);
        if (e == cudaSuccess) e = cudaEventRecord(L->ev_zready[s], L->stream);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(L->down_stream, L->ev_zready[s], 0);
        if (e == cudaSuccess) e = cudaMemcpyAsync(z_out_host, L->zs_async[s], zbytes, cudaMemcpyDeviceToHost, L->down_stream);
        if (e == cudaSuccess) e = cudaEventRecord(L->ev_down[s], L->down_stream);
    }
    if (e != cudaSuccess) return status_of(e);
    L->async_steps += 1;
    return SKIPCONV_OK;
}

// A pointer into pinned host memory that is mapped into the device's address space, as the device
// pointer of that same byte; NULL if the memory is not pinned and mapped.
static void* device_view(void* host)
{
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, host) != cudaSuccess || at.type != cudaMemoryTypeHost) {
        cudaGetLastError();
        return nullptr;
    }
    void* dev = nullptr;
    if (cudaHostGetDevicePointer(&dev, host, 0) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return dev;
}

int skipconv_step_host_sparse_async(skipconv_handle h, const void* x_t_host, float* z_blocks_host, int32_t* list_host,
                                    int32_t* count_host)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    if (!x_t_host || !z_blocks_host || !list_host || !count_host)
        return set_error("a host buffer is NULL"), SKIPCONV_ERR_INVALID;
    float* zb = static_cast<float*>(device_view(z_blocks_host));
    int32_t* lb = static_cast<int32_t*>(device_view(list_host));
    int32_t* cb = static_cast<int32_t*>(device_view(count_host));
    if (!zb || !lb || !cb)
        return set_error("the result buffers must be pinned host memory mapped into the device's address space"),
               SKIPCONV_ERR_INVALID;
    // upload and step as the pipelined call does, without the z read-back
    const int st = skipconv_step_host_async(h, x_t_host, nullptr);
    if (st) return st;
    // the step just enqueued used count slot (t - 1) % 2
    const cudaError_t e = launch_gather_open_blocks(*L, L->counters + ((L->t - 1) & 1), zb, lb, cb);
    return e == cudaSuccess ? SKIPCONV_OK : status_of(e);
}

int skipconv_sync(skipconv_handle h)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    // the copy streams exist once a pipelined call ran; the handle's stream may be the legacy default
    // stream (NULL), which is synchronised all the same
    cudaError_t e = L->up_stream ? cudaStreamSynchronize(L->up_stream) : cudaSuccess;
    if (e == cudaSuccess) e = cudaStreamSynchronize(L->stream);
    if (e == cudaSuccess && L->down_stream) e = cudaStreamSynchronize(L->down_stream);
    if (e != cudaSuccess) return status_of(e);
    return check_device_word(L);
}

int skipconv_destroy(skipconv_handle h)
{
    if (!h) return SKIPCONV_OK;
    Layer* L = get(h);
    {
        std::lock_guard<std::mutex> lock(live_mu());
        auto& v = live_layers();
        for (size_t i = 0; i < v.size();) {
            if (v[i] == L) {
                v[i] = v.back();
                v.pop_back();
                continue;
            }
            if (v[i]->link_x == L || v[i]->link_sc == L) v[i]->link_x = v[i]->link_sc = nullptr;
            ++i;
        }
    }
    cudaError_t e = cudaStreamSynchronize(L->stream);
    int st = e == cudaSuccess ? check_device_word(L) : status_of(e);
    async_release(L);
    free_buffers(L);
    delete h;
    return st;
}

int skipconv_get_z(skipconv_handle h, const float** z)
{
    Layer* L = get(h);
    if (!L || !z) return set_error("NULL argument"), SKIPCONV_ERR_INVALID;
    *z = L->z;
    return SKIPCONV_OK;
}

int skipconv_get_y(skipconv_handle h, const void** y)
{
    Layer* L = get(h);
    if (!L || !y) return set_error("NULL argument"), SKIPCONV_ERR_INVALID;
    *y = L->y;
    return SKIPCONV_OK;
}

int skipconv_get_prev_input(skipconv_handle h, const void** x_prev)
{
    Layer* L = get(h);
    if (!L || !x_prev) return set_error("NULL argument"), SKIPCONV_ERR_INVALID;
    *x_prev = L->xbuf[L->t & 1];
    return SKIPCONV_OK;
}

int skipconv_get_gate(skipconv_handle h, const uint8_t** block_mask, const int32_t** active_list,
                      const int32_t** active_count)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    if (block_mask) *block_mask = L->mask;
    if (active_list) *active_list = L->list;
    if (active_count) *active_count = L->counters + ((L->t + 1) & 1);  // slot of the last step (t - 1)
    return SKIPCONV_OK;
}

int skipconv_get_info(skipconv_handle h, skipconv_info* info)
{
    Layer* L = get(h);
    if (!L || !info) return set_error("NULL argument"), SKIPCONV_ERR_INVALID;
    info->ho = L->ho;
    info->wo = L->wo;
    info->nby = L->nby;
    info->nbx = L->nbx;
    info->conv_path = (L->fused == 2 && L->local_tc) ? SKIPCONV_PATH_TENSOR_CORE : L->path;
    info->fused = L->fused;
    info->num_sms = L->num_sms;
    info->state_bytes = L->state_bytes;
    return SKIPCONV_OK;
}

int skipconv_get_stats(skipconv_handle h, long long* active_blocks, long long* active_locations, double* macs)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    const size_t nblk = (size_t)L->p.n_streams * L->nby * L->nbx;
    uint8_t* m = (uint8_t*)malloc(nblk);
    if (!m) return set_error("host allocation failed"), SKIPCONV_ERR_OOM;
    cudaError_t e = cudaMemcpyAsync(m, L->mask, nblk, cudaMemcpyDeviceToHost, L->stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(L->stream);
    if (e != cudaSuccess) {
        free(m);
        return status_of(e);
    }
    long long nb = 0, nloc = 0;
    for (size_t k = 0; k < nblk; ++k) {
        if (!m[k]) continue;
        const int bx = (int)(k % L->nbx), by = (int)((k / L->nbx) % L->nby);
        const int bh = L->ho - by * L->p.block < L->p.block ? L->ho - by * L->p.block : L->p.block;
        const int bw = L->wo - bx * L->p.block < L->p.block ? L->wo - bx * L->p.block : L->p.block;
        ++nb;
        nloc += (long long)bh * bw;
    }
    free(m);
    if (active_blocks) *active_blocks = nb;
    if (active_locations) *active_locations = nloc;
    if (macs) *macs = (double)nloc * L->p.c_out * L->cpg * L->p.k_h * L->p.k_w;
    return check_device_word(L);
}

int skipconv_profile(skipconv_handle h, int enable)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    cudaError_t e = cudaStreamSynchronize(L->stream);
    if (e != cudaSuccess) return status_of(e);
    for (int k = 0; k < SKIPCONV_PROFILE_KINDS; ++k) {
        L->launches[k] = 0;
        L->prof_ms[k] = 0.0;
    }
    L->prof_n = 0;
    L->prof_on = enable ? 1 : 0;
    return SKIPCONV_OK;
}

int skipconv_profile_read(skipconv_handle h, long long* launches, double* ms)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    cudaError_t e = cudaStreamSynchronize(L->stream);
    if (e != cudaSuccess) return status_of(e);
    for (int i = 0; i < L->prof_n; ++i) {
        float t = 0.f;
        e = cudaEventElapsedTime(&t, L->prof_ev[2 * i], L->prof_ev[2 * i + 1]);
        if (e != cudaSuccess) return status_of(e);
        L->prof_ms[L->prof_kind[i]] += t;
    }
    L->prof_n = 0;
    for (int k = 0; k < SKIPCONV_PROFILE_KINDS; ++k) {
        if (launches) launches[k] = L->launches[k];
        if (ms) ms[k] = L->prof_ms[k];
    }
    return SKIPCONV_OK;
}

int skipconv_check_device(skipconv_handle h)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    cudaError_t e = cudaStreamSynchronize(L->stream);
    if (e != cudaSuccess) return status_of(e);
    return check_device_word(L);
}

namespace sc {
namespace {
// One bounded wait on a barrier that nothing completes: it runs out after limit_ns and records the timeout in
// the error word, the path every stuck wait of the library's kernels takes.
__global__ void selftest_wait_kernel(int* err, unsigned long long limit_ns)
{
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        ptx::mbar_init(ptx::smem_u32(&bar), 1);
        ptx::fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) ptx::mbar_wait(ptx::smem_u32(&bar), 0, nullptr, err, limit_ns);
}
}  // namespace
}  // namespace sc

int skipconv_selftest_timeout(skipconv_handle h, long long limit_ns)
{
    Layer* L = get(h);
    if (!L) return set_error("NULL handle"), SKIPCONV_ERR_INVALID;
    if (limit_ns < 1 || limit_ns > 1000000000LL)
        return set_error("limit_ns must be in 1 .. 1e9"), SKIPCONV_ERR_INVALID;
    if (int st = check_device_word(L)) return st;
    selftest_wait_kernel<<<1, 32, 0, L->stream>>>(L->err_dev, (unsigned long long)limit_ns);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) e = cudaStreamSynchronize(L->stream);
    if (e != cudaSuccess) return status_of(e);
    return check_device_word(L);
}

}  // extern "C"
