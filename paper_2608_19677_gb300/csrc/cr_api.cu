// Context, scratch memory and status handling of the C ABI (include/cacheroute.h).
#include <stdlib.h>
#include <string.h>

#include <cuda.h>

#include "cr_internal.cuh"

static char g_create_msg[320] = "no error";

int cr_fail(cr_ctx *ctx, int code, const char *fmt, ...)
{
    char *dst = ctx ? ctx->msg : g_create_msg;
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(dst, 320, fmt, ap);
    va_end(ap);
    return code;
}

int cr_check_launch(cr_ctx *ctx, const char *what)
{
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return cr_fail(ctx, CR_ECUDA, "launch of %s failed: %s", what, cudaGetErrorString(e));
    return CR_OK;
}

int cr_scratch(cr_ctx *ctx, int slot, size_t bytes, void **out)
{
    if (bytes == 0) bytes = 16;
    if (ctx->scratch_bytes[slot] < bytes) {
        if (ctx->scratch[slot]) {
            // the old buffer may still be read by enqueued work
            cudaError_t e = cudaStreamSynchronize(ctx->stream);
            if (e != cudaSuccess) return cr_fail(ctx, CR_ECUDA, "scratch sync: %s", cudaGetErrorString(e));
            cudaFree(ctx->scratch[slot]);
            ctx->scratch[slot] = NULL;
            ctx->scratch_bytes[slot] = 0;
        }
        size_t grow = bytes + bytes / 4;
        grow = (grow + 255) & ~(size_t)255;
        void *p = NULL;
        if (cudaMalloc(&p, grow) != cudaSuccess) {
            cudaGetLastError();
            return cr_fail(ctx, CR_ENOMEM, "scratch slot %d: cannot allocate %zu bytes", slot, grow);
        }
        ctx->scratch[slot] = p;
        ctx->scratch_bytes[slot] = grow;
    }
    *out = ctx->scratch[slot];
    return CR_OK;
}

extern "C" int cr_create(cr_ctx **out, int device, void *cuda_stream)
{
    if (!out) return cr_fail(NULL, CR_EINVAL, "cr_create: out is NULL");
    *out = NULL;
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev) {
        cudaGetLastError();
        return cr_fail(NULL, CR_EINVAL, "cr_create: device %d not available (%d devices)", device, ndev);
    }
    if (cudaSetDevice(device) != cudaSuccess) {
        cudaGetLastError();
        return cr_fail(NULL, CR_ECUDA, "cr_create: cudaSetDevice(%d) failed", device);
    }
    cr_ctx *c = (cr_ctx *)calloc(1, sizeof(cr_ctx));
    if (!c) return cr_fail(NULL, CR_ENOMEM, "cr_create: host allocation failed");
    c->device = device;
    c->stream = (cudaStream_t)cuda_stream;
    cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, device);
    if (c->num_sms <= 0) c->num_sms = 1;
    if (cudaMalloc(&c->d_status, sizeof(uint32_t)) != cudaSuccess ||
        cudaMemset(c->d_status, 0, sizeof(uint32_t)) != cudaSuccess) {
        cudaGetLastError();
        free(c);
        return cr_fail(NULL, CR_ENOMEM, "cr_create: status word allocation failed");
    }
    strcpy(c->msg, "no error");
    *out = c;
    return CR_OK;
}

static void prof_free(cr_ctx *ctx)
{
    cr_prof &P = ctx->prof;
    if (P.ev) {
        for (uint32_t i = 0; i < 2 * P.cap; ++i)
            if (P.ev[i]) cudaEventDestroy(P.ev[i]);
        free(P.ev);
    }
    free(P.tag);
    memset(&P, 0, sizeof(P));
}

extern "C" int cr_profile_enable(cr_ctx *ctx, uint32_t max_launches)
{
    if (!ctx) return CR_EINVAL;
    CR_CUDA(ctx, cudaStreamSynchronize(ctx->stream));
    if (ctx->resolve_stream) CR_CUDA(ctx, cudaStreamSynchronize(ctx->resolve_stream));
    if (max_launches == ctx->prof.cap && ctx->prof.ev) {  // same size: keep the events, forget the launches
        ctx->prof.used = 0;
        return CR_OK;
    }
    prof_free(ctx);
    if (max_launches == 0) return CR_OK;
    cr_prof &P = ctx->prof;
    P.ev = (cudaEvent_t *)calloc(2 * (size_t)max_launches, sizeof(cudaEvent_t));
    P.tag = (uint8_t *)calloc(max_launches, 1);
    if (!P.ev || !P.tag) {
        prof_free(ctx);
        return cr_fail(ctx, CR_ENOMEM, "cr_profile_enable: host allocation failed");
    }
    P.cap = max_launches;
    for (uint32_t i = 0; i < 2 * max_launches; ++i) {
        if (cudaEventCreate(&P.ev[i]) != cudaSuccess) {
            cudaGetLastError();
            prof_free(ctx);
            return cr_fail(ctx, CR_ECUDA, "cr_profile_enable: cannot create events");
        }
    }
    return CR_OK;
}

extern "C" int cr_profile_read(cr_ctx *ctx, uint32_t tag, uint64_t *launches, double *total_ms)
{
    if (!ctx || !launches || !total_ms) return CR_EINVAL;
    if (tag >= CR_PROF_TAGS) return cr_fail(ctx, CR_EINVAL, "cr_profile_read: tag %u", tag);
    uint64_t n = 0;
    double ms = 0.0;
    const cr_prof &P = ctx->prof;
    for (uint32_t i = 0; i < P.used; ++i) {
        if (P.tag[i] != tag) continue;
        CR_CUDA(ctx, cudaEventSynchronize(P.ev[2 * i + 1]));
        float x = 0.f;
        CR_CUDA(ctx, cudaEventElapsedTime(&x, P.ev[2 * i], P.ev[2 * i + 1]));
        ms += x;
        ++n;
    }
    *launches = n;
    *total_ms = ms;
    return CR_OK;
}

extern "C" int cr_destroy(cr_ctx *ctx)
{
    if (!ctx) return CR_OK;
    cudaStreamSynchronize(ctx->stream);
    prof_free(ctx);
    cr_replay_input_destroy(nullptr, ctx->replay_in);
    if (ctx->resolve_stream) cudaStreamSynchronize(ctx->resolve_stream);
    if (ctx->ev_cand) cudaEventDestroy(ctx->ev_cand);
    if (ctx->ev_resolve) cudaEventDestroy(ctx->ev_resolve);
    for (int i = 0; i < SCR_NUM; ++i)
        if (ctx->scratch[i]) cudaFree(ctx->scratch[i]);
    cudaFree(ctx->d_status);
    free(ctx);
    return CR_OK;
}

extern "C" int cr_set_stream(cr_ctx *ctx, void *cuda_stream)
{
    if (!ctx) return CR_EINVAL;
    ctx->stream = (cudaStream_t)cuda_stream;
    return CR_OK;
}

extern "C" int cr_set_resolve_stream(cr_ctx *ctx, void *cuda_stream)
{
    if (!ctx) return CR_EINVAL;
    if (cuda_stream && !ctx->ev_cand) {
        CR_CUDA(ctx, cudaEventCreateWithFlags(&ctx->ev_cand, cudaEventDisableTiming));
        CR_CUDA(ctx, cudaEventCreateWithFlags(&ctx->ev_resolve, cudaEventDisableTiming));
    }
    if (ctx->resolve_stream == (cudaStream_t)cuda_stream) return CR_OK;  // unchanged: keep the ordering state
    if (ctx->resolve_stream) CR_CUDA(ctx, cudaStreamSynchronize(ctx->resolve_stream));
    ctx->resolve_stream = (cudaStream_t)cuda_stream;
    ctx->resolve_recorded = 0;  // the old stream's work is finished
    return CR_OK;
}

// ---- SM partition (green contexts, reached through the runtime's driver entry points) ----
struct cr_partition {
    CUgreenCtx g[2];
    CUstream s[2];
};

template <typename F>
static int driver_fn(const char *name, F *fp)
{
    cudaDriverEntryPointQueryResult q;
    void *p = nullptr;
    if (cudaGetDriverEntryPointByVersion(name, &p, CUDART_VERSION, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !p) {
        cudaGetLastError();
        return CR_ECUDA;
    }
    *fp = reinterpret_cast<F>(p);
    return CR_OK;
}

typedef CUresult (*fDeviceGet)(CUdevice *, int);
typedef CUresult (*fGetRes)(CUdevice, CUdevResource *, CUdevResourceType);
typedef CUresult (*fSplit)(CUdevResource *, unsigned int *, const CUdevResource *, CUdevResource *, unsigned int,
                           unsigned int);
typedef CUresult (*fDesc)(CUdevResourceDesc *, CUdevResource *, unsigned int);
typedef CUresult (*fGreen)(CUgreenCtx *, CUdevResourceDesc, CUdevice, unsigned int);
typedef CUresult (*fStream)(CUstream *, CUgreenCtx, unsigned int, int);

static int partition_create(int device, uint32_t small_sms, cr_partition **out, void **big_stream,
                            void **small_stream);

extern "C" int cr_partition_create(int device, uint32_t small_sms, cr_partition **out, void **big_stream,
                                   void **small_stream)
{
    if (!out || !big_stream || !small_stream) return cr_fail(NULL, CR_EINVAL, "cr_partition_create: NULL output");
    *out = nullptr;
    int prev_dev = -1;
    if (cudaGetDevice(&prev_dev) != cudaSuccess) {
        cudaGetLastError();
        prev_dev = -1;
    }
    const int st = partition_create(device, small_sms, out, big_stream, small_stream);
    if (prev_dev >= 0) cudaSetDevice(prev_dev);  // the caller's current device is left as it was
    return st;
}

static int partition_create(int device, uint32_t small_sms, cr_partition **out, void **big_stream,
                            void **small_stream)
{
    fDeviceGet deviceGet;
    fGetRes getRes;
    fSplit split;
    fDesc desc;
    fGreen green;
    fStream stream;
    if (cudaSetDevice(device) != cudaSuccess || cudaFree(0) != cudaSuccess) {
        cudaGetLastError();
        return cr_fail(NULL, CR_EINVAL, "cr_partition_create: device %d not available", device);
    }
    if (driver_fn("cuDeviceGet", &deviceGet) || driver_fn("cuDeviceGetDevResource", &getRes) ||
        driver_fn("cuDevSmResourceSplitByCount", &split) || driver_fn("cuDevResourceGenerateDesc", &desc) ||
        driver_fn("cuGreenCtxCreate", &green) || driver_fn("cuGreenCtxStreamCreate", &stream))
        return cr_fail(NULL, CR_ECUDA, "cr_partition_create: green contexts are not available from this driver");
    CUdevice dev;
    CUdevResource sm, part, rest;
    if (deviceGet(&dev, device) != CUDA_SUCCESS || getRes(dev, &sm, CU_DEV_RESOURCE_TYPE_SM) != CUDA_SUCCESS)
        return cr_fail(NULL, CR_ECUDA, "cr_partition_create: cannot read the SM resource");
    if (small_sms == 0 || small_sms >= sm.sm.smCount)
        return cr_fail(NULL, CR_EINVAL, "cr_partition_create: small_sms=%u outside 1..%u", small_sms,
                       sm.sm.smCount - 1);
    unsigned int nb = 1;
    if (split(&part, &nb, &sm, &rest, 0, sm.sm.smCount - small_sms) != CUDA_SUCCESS || nb != 1 ||
        rest.sm.smCount == 0)
        return cr_fail(NULL, CR_ECUDA, "cr_partition_create: cannot split %u SMs", sm.sm.smCount);
    cr_partition *pt = (cr_partition *)calloc(1, sizeof(cr_partition));
    if (!pt) return cr_fail(NULL, CR_ENOMEM, "cr_partition_create: host allocation failed");
    CUdevResource *res[2] = {&part, &rest};
    for (int i = 0; i < 2; ++i) {
        CUdevResourceDesc d;
        if (desc(&d, res[i], 1) != CUDA_SUCCESS || green(&pt->g[i], d, dev, CU_GREEN_CTX_DEFAULT_STREAM) != CUDA_SUCCESS ||
            stream(&pt->s[i], pt->g[i], CU_STREAM_NON_BLOCKING, 0) != CUDA_SUCCESS) {
            cr_partition_destroy(pt);
            return cr_fail(NULL, CR_ECUDA, "cr_partition_create: cannot create the green context");
        }
    }
    *out = pt;
    *big_stream = (void *)pt->s[0];
    *small_stream = (void *)pt->s[1];
    return CR_OK;
}

extern "C" int cr_partition_destroy(cr_partition *pt)
{
    if (!pt) return CR_OK;
    typedef CUresult (*fStreamDestroy)(CUstream);
    typedef CUresult (*fGreenDestroy)(CUgreenCtx);
    fStreamDestroy sd = nullptr;
    fGreenDestroy gd = nullptr;
    driver_fn("cuStreamDestroy", &sd);
    driver_fn("cuGreenCtxDestroy", &gd);
    for (int i = 0; i < 2; ++i) {
        if (pt->s[i] && sd) {
            cudaStreamSynchronize((cudaStream_t)pt->s[i]);
            sd(pt->s[i]);
        }
        if (pt->g[i] && gd) gd(pt->g[i]);
    }
    free(pt);
    return CR_OK;
}

extern "C" int cr_sync(cr_ctx *ctx)
{
    if (!ctx) return CR_EINVAL;
    CR_CUDA(ctx, cudaStreamSynchronize(ctx->stream));
    // a split route call's resolution raises its flags on the resolve stream:
    // wait for it too, so that no flag is missed or reported against a later call
    if (ctx->resolve_stream && ctx->resolve_recorded) CR_CUDA(ctx, cudaEventSynchronize(ctx->ev_resolve));
    uint32_t flags = 0;
    CR_CUDA(ctx, cudaMemcpy(&flags, ctx->d_status, sizeof(flags), cudaMemcpyDeviceToHost));
    if (flags) {
        CR_CUDA(ctx, cudaMemset(ctx->d_status, 0, sizeof(uint32_t)));
        if (flags & CR_FLAG_BADDEST)
            return cr_fail(ctx, CR_EINVAL, "a destination index >= R reached the replay (skipped)");
        if (flags & CR_FLAG_OVERFLOW)
            return cr_fail(ctx, CR_EOVERFLOW, "a load or counter exceeded its documented range");
        if (flags & CR_FLAG_TIMEOUT)
            return cr_fail(ctx, CR_ETIMEOUT, "a bounded device-side wait gave up");
        if (flags & CR_FLAG_BOUNDS)
            return cr_fail(ctx, CR_EINVAL, "debug build: an index outside its array was skipped (results of that "
                                           "call are not meaningful)");
        if (flags & CR_FLAG_INTERNAL)
            return cr_fail(ctx, CR_ECUDA, "a kernel found its state inconsistent (results of that call are not "
                                          "meaningful)");
        if (flags & CR_FLAG_BADSIZE)
            return cr_fail(ctx, CR_EINVAL,
                           "token-weighted replay: a key came back with another prefix length (counters of "
                           "that call are not meaningful)");
    }
    return CR_OK;
}

extern "C" const char *cr_last_error(const cr_ctx *ctx)
{
    return ctx ? ctx->msg : g_create_msg;
}

extern "C" uint64_t cr_launch_count(const cr_ctx *ctx)
{
    return ctx ? ctx->launches : 0;
}
