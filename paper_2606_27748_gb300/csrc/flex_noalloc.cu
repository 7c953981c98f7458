// flex_linattn_bwd_noalloc: the backward entry point for callers that cannot allocate
// device memory and so cannot hand the library a workspace.
//
// It always runs the fp32 CUDA-core (SIMT) backward, whose only scratch is the
// per-sequence partial frequency gradients (B * H * (Mc * d + 1) floats, Mc = M or 2M)
// before they are summed over the batch; the tensor-core backward's scratch (dW partials
// of 128 rows per frequency group, pass and sequence, plus key weights growing with N) is
// several times larger.  Here that scratch is a
// fixed array in the library's own device memory instead, so nothing is allocated per
// call: every GPU that loads the library holds the array (4 MiB) until the process exits.
#include <cuda.h>

#include "flex_internal.h"

#include <mutex>

namespace {

constexpr size_t kNoallocScratchFloats = (size_t)1 << 20;  // 4 MiB of fp32

// The scratch.  In host code this name is only a stand-in for the device symbol, never a
// usable address: the device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) float g_bwd_scratch[kNoallocScratchFloats];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
// Per device: the unique id of the context the address was looked up in, and the
// address.  A device's module (and with it the array) is reloaded in a new context, e.g.
// after cudaDeviceReset, and may land at another address, so a new context forces a new
// lookup.  Context ids are never reused within a process (a context handle may be).
unsigned long long g_scratch_ctx_id[kMaxDevices] = {};
float* g_scratch_ptr[kMaxDevices] = {};

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

void* driver_fn(const char* name)
{
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion(name, &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
        return nullptr;
    return p;
}

// Id of the current context (0 if none is current).
int current_ctx_id(unsigned long long* id)
{
    static CtxGetCurrentFn get = (CtxGetCurrentFn)driver_fn("cuCtxGetCurrent");
    static CtxGetIdFn get_id = (CtxGetIdFn)driver_fn("cuCtxGetId");
    CUcontext ctx = nullptr;
    *id = 0;
    if (!get || !get_id || get(&ctx) != CUDA_SUCCESS) return FLEX_ECUDA;
    if (ctx && get_id(ctx, id) != CUDA_SUCCESS) return FLEX_ECUDA;
    return FLEX_OK;
}

// Device address of g_bwd_scratch on the current device, looked up (with the device
// current) once per device and context.
int scratch_for_current_device(float** out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return FLEX_ECUDA;
    if (dev < 0 || dev >= kMaxDevices) return FLEX_EUNSUPPORTED;
    unsigned long long id = 0;
    if (current_ctx_id(&id) != FLEX_OK) return FLEX_ECUDA;
    std::lock_guard<std::mutex> lock(g_mu);
    if (id == 0 || !g_scratch_ptr[dev] || g_scratch_ctx_id[dev] != id) {
        // (the lookup also creates the device's primary context if none is current yet)
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_bwd_scratch) != cudaSuccess || p == nullptr)
            return FLEX_ECUDA;
        if (current_ctx_id(&id) != FLEX_OK || id == 0) return FLEX_ECUDA;
        g_scratch_ptr[dev] = static_cast<float*>(p);
        g_scratch_ctx_id[dev] = id;
    }
    *out = g_scratch_ptr[dev];
    return FLEX_OK;
}

}  // namespace

extern "C" int flex_linattn_bwd_noalloc(const flex_shape* shape, const void* q, const void* k,
                                        const void* v, const float* W1, const float* W2,
                                        int causal, const void* out, const float* den,
                                        const void* dout, void* dq, void* dk, void* dv,
                                        float* dW1, float* dW2, void* stream)
{
    if (!shape) return FLEX_EINVAL;
    if (shape->B < 1 || shape->H < 1 || shape->N < 1 || shape->d < 1 || shape->M < 1)
        return FLEX_EINVAL;
    if (shape->dtype != FLEX_F32 && shape->dtype != FLEX_BF16) return FLEX_EINVAL;
    if (shape->d > 128 || shape->M > 256 || shape->d % 4 != 0) return FLEX_EUNSUPPORTED;
    if (!q || !k || !v || !W1 || !out || !den || !dout || !dq || !dk || !dv || !dW1)
        return FLEX_EINVAL;
    if ((W2 == nullptr) != (dW2 == nullptr)) return FLEX_EINVAL;
    for (const void* t : {q, k, v, (const void*)W1, out, (const void*)den, dout, (const void*)dq,
                          (const void*)dk, (const void*)dv, (const void*)dW1, (const void*)W2,
                          (const void*)dW2})
        if (t && ((uintptr_t)t % 16) != 0) return FLEX_EINVAL;

    flex::Problem p;
    p.B = shape->B; p.H = shape->H; p.N = shape->N; p.d = shape->d; p.M = shape->M;
    p.bf16 = shape->dtype == FLEX_BF16;
    p.nonstat = W2 != nullptr;
    p.causal = causal ? 1 : 0;
    if (flex::simt_pick_chunk_bwd(p) == 0) return FLEX_EUNSUPPORTED;
    // The fixed scratch must hold every partial; larger problems are refused.
    if (flex::simt_bwd_ws_bytes(p) > kNoallocScratchFloats * sizeof(float))
        return FLEX_EWORKSPACE;

    float* scratch = nullptr;
    int rc = scratch_for_current_device(&scratch);
    if (rc != FLEX_OK) return rc;
    // Every partial slot the reduction reads is written first by this call, so the
    // array's previous contents need no clearing.
    cudaError_t e = flex::launch_simt_bwd(p, q, k, v, W1, W2, nullptr, out, den, dout, dq, dk,
                                          dv, dW1, dW2, nullptr, scratch, (cudaStream_t)stream);
    if (e != cudaSuccess) return FLEX_ECUDA;
    flex::add_launches(2);  // the SIMT backward and its dW reduction
    return FLEX_OK;
}
