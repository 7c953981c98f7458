// Host side of the C ABI declared in include/flexattn.h: argument validation, workspace
// layout and kernel dispatch.  Nothing here allocates device memory or synchronises,
// except flex_check_status.
#include "flex_internal.h"

#include <stdint.h>

#include <algorithm>
#include <atomic>

using flex::Problem;

namespace {

bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

// Fills `p` from `s`; FLEX_OK or the error to return.
int make_problem(const flex_shape* s, const float* W2, int causal, Problem* p)
{
    if (!s) return FLEX_EINVAL;
    if (s->B < 1 || s->H < 1 || s->N < 1 || s->d < 1 || s->M < 1) return FLEX_EINVAL;
    if (s->dtype != FLEX_F32 && s->dtype != FLEX_BF16) return FLEX_EINVAL;
    if ((long long)s->B * s->H > (1LL << 30)) return FLEX_EUNSUPPORTED;
    if ((long long)s->N > (1LL << 30)) return FLEX_EUNSUPPORTED;
    if (s->d > 128 || s->M > 256 || s->d % 4 != 0) return FLEX_EUNSUPPORTED;
    p->B = s->B; p->H = s->H; p->N = s->N; p->d = s->d; p->M = s->M;
    p->bf16 = s->dtype == FLEX_BF16;
    p->nonstat = W2 != nullptr;
    p->causal = causal ? 1 : 0;
    return FLEX_OK;
}

size_t header_bytes() { return sizeof(flex::WsHeader); }

int check_ws(void* ws, size_t ws_bytes, size_t need)
{
    if (!ws) return FLEX_EINVAL;
    if (!aligned(ws, 256)) return FLEX_EINVAL;
    if (ws_bytes < need) return FLEX_EWORKSPACE;
    return FLEX_OK;
}

// Header, the non-causal partial states (tensor-core path), then the key weights of the
// norm prefactor [B*H*N] fp32 (tensor-core paths, used only when tau is given).
size_t nc_scratch_bytes(const Problem& p)
{
    return flex::tc_nc_supported(p) ? flex::align_up(flex::tc_nc_ws_bytes(p), 256) : 0;
}
size_t kw_bytes(const Problem& p)
{
    const bool tc = flex::tc_fwd_supported(p) || flex::tc_nc_supported(p);
    return tc ? flex::align_up((size_t)p.B * p.H * p.N * sizeof(float), 256) : 0;
}
size_t fwd_ws_bytes(const Problem& p) { return header_bytes() + nc_scratch_bytes(p) + kw_bytes(p); }

size_t bwd_ws_bytes(const Problem& p)
{
    size_t scratch = flex::simt_bwd_ws_bytes(p);
    if (flex::tc_bwd_supported(p)) scratch = std::max(scratch, flex::tc_bwd_ws_bytes(p));
    return header_bytes() + flex::align_up(scratch, 256);
}

std::atomic<unsigned long long> g_launches{0};

// Records `n` enqueued kernels when the launch sequence succeeded.
int count(int n, cudaError_t e)
{
    if (e != cudaSuccess) return FLEX_ECUDA;
    g_launches += (unsigned long long)n;
    return FLEX_OK;
}

}  // namespace

void flex::add_launches(int n) { g_launches += (unsigned long long)n; }

extern "C" {

const char* flex_strerror(int status)
{
    switch (status) {
    case FLEX_OK: return "ok";
    case FLEX_EINVAL: return "invalid argument (null/misaligned pointer, bad shape or W2/dW2 mismatch)";
    case FLEX_EUNSUPPORTED: return "unsupported shape or dtype";
    case FLEX_EWORKSPACE: return "workspace too small";
    case FLEX_ECUDA: return "CUDA error";
    case FLEX_ETIMEOUT: return "a device-side bounded wait gave up";
    default: return "unknown status";
    }
}

size_t flex_workspace_bytes(const flex_shape* shape, int causal, int backward)
{
    Problem p;
    if (make_problem(shape, nullptr, causal, &p) != FLEX_OK) return 0;
    // Size for the larger of the two variants' scratch.
    p.nonstat = 1;
    return backward ? bwd_ws_bytes(p) : fwd_ws_bytes(p);
}

int flex_featmap(const flex_shape* shape, const void* x, const float* W1, const float* W2,
                 void* phi, void* stream)
{
    Problem p;
    int rc = make_problem(shape, W2, 0, &p);
    if (rc) return rc;
    if (!x || !W1 || !phi) return FLEX_EINVAL;
    if (!aligned(x, 16) || !aligned(W1, 16) || !aligned(phi, 16) || (W2 && !aligned(W2, 16)))
        return FLEX_EINVAL;
    if (flex::tc_featmap_supported(p))  // tensor-core projection (no workspace: no status)
        return count(1, flex::launch_tc_featmap(p, x, W1, W2, nullptr, phi, nullptr,
                                                (cudaStream_t)stream));
    return count(1, flex::launch_featmap(p, x, W1, W2, phi, (cudaStream_t)stream));
}

int flex_linattn_fwd(const flex_shape* shape, const void* q, const void* k, const void* v,
                     const float* W1, const float* W2, const float* tau, int causal, void* out,
                     float* den, void* ws, size_t ws_bytes, void* stream)
{
    Problem p;
    int rc = make_problem(shape, W2, causal, &p);
    if (rc) return rc;
    if (!q || !k || !v || !W1 || !out) return FLEX_EINVAL;
    for (const void* t : {q, k, v, (const void*)W1, (const void*)out})
        if (!aligned(t, 16)) return FLEX_EINVAL;
    if ((W2 && !aligned(W2, 16)) || (den && !aligned(den, 16)) || (tau && !aligned(tau, 4)))
        return FLEX_EINVAL;
    if ((rc = check_ws(ws, ws_bytes, fwd_ws_bytes(p)))) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    int* status = &((flex::WsHeader*)ws)->status;
    const bool tcf = flex::tc_fwd_supported(p), tcn = !tcf && flex::tc_nc_supported(p);
    if (tcf || tcn) {
        float* kw = nullptr;  // key weights of the norm prefactor, one pass over k
        if (tau) {
            kw = (float*)((char*)ws + header_bytes() + nc_scratch_bytes(p));
            if (int e = count(1, flex::launch_key_weights(p, k, tau, kw, s))) return e;
        }
        if (tcf) return count(1, flex::launch_tc_fwd(p, q, k, v, W1, W2, kw, out, den, status, s));
        return count(3, flex::launch_tc_nc(p, q, k, v, W1, W2, kw, out, den,
                                           (char*)ws + header_bytes(), status, s));
    }
    if (flex::simt_pick_chunk_fwd(p) == 0) return FLEX_EUNSUPPORTED;
    return count(1, flex::launch_simt_fwd(p, q, k, v, W1, W2, tau, out, den, s));
}

int flex_linattn_bwd(const flex_shape* shape, const void* q, const void* k, const void* v,
                     const float* W1, const float* W2, const float* tau, int causal,
                     const void* out, const float* den, const void* dout, void* dq, void* dk,
                     void* dv, float* dW1, float* dW2, float* dtau, void* ws, size_t ws_bytes,
                     void* stream)
{
    Problem p;
    int rc = make_problem(shape, W2, causal, &p);
    if (rc) return rc;
    if (!q || !k || !v || !W1 || !out || !den || !dout || !dq || !dk || !dv || !dW1)
        return FLEX_EINVAL;
    if ((W2 == nullptr) != (dW2 == nullptr) || (tau == nullptr) != (dtau == nullptr))
        return FLEX_EINVAL;
    if ((tau && !aligned(tau, 4)) || (dtau && !aligned(dtau, 4))) return FLEX_EINVAL;
    for (const void* t : {q, k, v, (const void*)W1, out, (const void*)den, dout, (const void*)dq,
                          (const void*)dk, (const void*)dv, (const void*)dW1})
        if (!aligned(t, 16)) return FLEX_EINVAL;
    if ((W2 && !aligned(W2, 16)) || (dW2 && !aligned(dW2, 16))) return FLEX_EINVAL;
    if ((rc = check_ws(ws, ws_bytes, bwd_ws_bytes(p)))) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    void* scratch = (char*)ws + header_bytes();
    if (flex::tc_bwd_supported(p))  // with tau: one more launch, the key weights
        return count(flex::tc_bwd_launches(p, tau != nullptr),
                     flex::launch_tc_bwd(p, q, k, v, W1, W2, tau, out, den, dout, dq, dk, dv,
                                         dW1, dW2, dtau, scratch, &((flex::WsHeader*)ws)->status,
                                         s));
    if (flex::simt_pick_chunk_bwd(p) == 0) return FLEX_EUNSUPPORTED;
    return count(2, flex::launch_simt_bwd(p, q, k, v, W1, W2, tau, out, den, dout, dq, dk, dv,
                                          dW1, dW2, dtau, scratch, s));
}

size_t flex_decode_workspace_bytes(const flex_shape* shape)
{
    Problem p;
    if (make_problem(shape, nullptr, 1, &p) != FLEX_OK || p.N != 1) return 0;
    return header_bytes() + flex::align_up(flex::decode_ws_bytes(p), 256);
}

int flex_linattn_decode(const flex_shape* shape, const void* q, const void* k, const void* v,
                        const float* W1, const float* W2, const float* tau, float* S, float* z,
                        void* out, float* den, void* ws, size_t ws_bytes, void* stream)
{
    Problem p;
    int rc = make_problem(shape, W2, 1, &p);
    if (rc) return rc;
    if (p.N != 1) return FLEX_EINVAL;
    if (!q || !k || !v || !W1 || !S || !z || !out) return FLEX_EINVAL;
    for (const void* t : {q, k, v, (const void*)W1, (const void*)S, (const void*)z, (const void*)out})
        if (!aligned(t, 16)) return FLEX_EINVAL;
    if ((W2 && !aligned(W2, 16)) || (den && !aligned(den, 16)) || (tau && !aligned(tau, 4)))
        return FLEX_EINVAL;
    if ((rc = check_ws(ws, ws_bytes, header_bytes() + flex::decode_ws_bytes(p)))) return rc;
    return count(2, flex::launch_decode(p, q, k, v, W1, W2, tau, S, z, out, den,
                                        (char*)ws + header_bytes(),
                                        &((flex::WsHeader*)ws)->status, (cudaStream_t)stream));
}

// Distillation-loss workspace: header, phi(q), phi~(k) [B*H*N][2M] bf16, key weights
// [B*H*N] fp32, partial sums [B*H][query blocks] fp32; for the gradient also the row
// statistics [B*H*N] float4, the dW slots and the dtau partials [2*B*H] fp32.
struct AwdWs {
    size_t pq, pk, kw, part, rowstat, slots, dtau_part, total;
};
AwdWs awd_ws(const Problem& p, bool grad)
{
    const size_t rows = (size_t)p.B * p.H * p.N, feat = flex::align_up(rows * 2 * p.M * 2, 256);
    AwdWs w;
    w.pq = header_bytes();
    w.pk = w.pq + feat;
    w.kw = w.pk + feat;
    w.part = w.kw + flex::align_up(rows * sizeof(float), 256);
    w.rowstat = w.part + flex::align_up(flex::tc_awd_part_floats(p) * sizeof(float), 256);
    w.slots = w.rowstat + (grad ? flex::align_up(rows * 16, 256) : 0);
    w.dtau_part = w.slots + (grad ? flex::align_up(flex::tc_awd_slot_floats(p) * 4, 256) : 0);
    w.total = w.dtau_part + (grad ? flex::align_up((size_t)2 * p.B * p.H * 4, 256) : 0);
    return w;
}

size_t flex_awd_workspace_bytes(const flex_shape* shape)
{
    Problem p;
    if (make_problem(shape, nullptr, 0, &p) != FLEX_OK || !flex::tc_awd_supported(p)) return 0;
    return awd_ws(p, false).total;
}

int flex_awd_loss(const flex_shape* shape, const void* q, const void* k, const float* W1,
                  const float* W2, const float* tau, int causal, float* loss, void* ws,
                  size_t ws_bytes, void* stream)
{
    Problem p;
    int rc = make_problem(shape, W2, causal, &p);
    if (rc) return rc;
    if (!q || !k || !W1 || !loss) return FLEX_EINVAL;
    for (const void* t : {q, k, (const void*)W1, (const void*)loss})
        if (!aligned(t, 16)) return FLEX_EINVAL;
    if ((W2 && !aligned(W2, 16)) || (tau && !aligned(tau, 4))) return FLEX_EINVAL;
    if (!flex::tc_awd_supported(p)) return FLEX_EUNSUPPORTED;
    const AwdWs w = awd_ws(p, false);
    if ((rc = check_ws(ws, ws_bytes, w.total))) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    char* base = (char*)ws;
    float* kw = tau ? (float*)(base + w.kw) : nullptr;
    if (tau && (rc = count(1, flex::launch_key_weights(p, k, tau, kw, s)))) return rc;
    int* status = &((flex::WsHeader*)ws)->status;
    if ((rc = count(1, flex::launch_tc_featmap(p, q, W1, W2, nullptr, base + w.pq, status, s))))
        return rc;
    if ((rc = count(1, flex::launch_tc_featmap(p, k, W1, W2, kw, base + w.pk, status, s))))
        return rc;
    return count(2, flex::launch_tc_awd(p, q, k, base + w.pq, base + w.pk, (float*)(base + w.part),
                                        loss, status, s));
}

size_t flex_awd_bwd_workspace_bytes(const flex_shape* shape)
{
    Problem p;
    if (make_problem(shape, nullptr, 0, &p) != FLEX_OK || !flex::tc_awd_supported(p)) return 0;
    return awd_ws(p, true).total;
}

int flex_awd_loss_bwd(const flex_shape* shape, const void* q, const void* k, const float* W1,
                      const float* W2, const float* tau, int causal, const float* dloss,
                      float* loss, float* dW1, float* dW2, float* dtau, void* ws,
                      size_t ws_bytes, void* stream)
{
    Problem p;
    int rc = make_problem(shape, W2, causal, &p);
    if (rc) return rc;
    if (!q || !k || !W1 || !dloss || !dW1) return FLEX_EINVAL;
    if ((W2 != nullptr) != (dW2 != nullptr) || (tau != nullptr) != (dtau != nullptr))
        return FLEX_EINVAL;
    for (const void* t : {q, k, (const void*)W1, (const void*)dW1})
        if (!aligned(t, 16)) return FLEX_EINVAL;
    if ((W2 && (!aligned(W2, 16) || !aligned(dW2, 16))) || (tau && !aligned(tau, 4)) ||
        (loss && !aligned(loss, 4)) || !aligned(dloss, 4) || (dtau && !aligned(dtau, 4)))
        return FLEX_EINVAL;
    if (!flex::tc_awd_supported(p)) return FLEX_EUNSUPPORTED;
    const AwdWs w = awd_ws(p, true);
    if ((rc = check_ws(ws, ws_bytes, w.total))) return rc;
    cudaStream_t s = (cudaStream_t)stream;
    char* base = (char*)ws;
    float* kw = tau ? (float*)(base + w.kw) : nullptr;
    if (tau && (rc = count(1, flex::launch_key_weights(p, k, tau, kw, s)))) return rc;
    int* status = &((flex::WsHeader*)ws)->status;
    if ((rc = count(1, flex::launch_tc_featmap(p, q, W1, W2, nullptr, base + w.pq, status, s))))
        return rc;
    if ((rc = count(1, flex::launch_tc_featmap(p, k, W1, W2, kw, base + w.pk, status, s))))
        return rc;
    return count(loss ? 4 : 3,
                 flex::launch_tc_awd_bwd(p, q, k, base + w.pq, base + w.pk, W1, W2, kw, tau, dloss,
                                         (float*)(base + w.part), loss,
                                         (float4*)(base + w.rowstat), (float*)(base + w.slots),
                                         (float*)(base + w.dtau_part), dW1, dW2, dtau, status, s));
}

unsigned long long flex_kernel_launches(void) { return g_launches.load(); }

int flex_debug_stall(void* ws, size_t ws_bytes, int cycles, void* stream)
{
    if (!ws || !aligned(ws, 256) || cycles < 0) return FLEX_EINVAL;
    if (ws_bytes < header_bytes()) return FLEX_EWORKSPACE;
    // from pageable host memory: the value is staged before the call returns
    int* word = (int*)ws + flex::kStallWord;
    return cudaMemcpyAsync(word, &cycles, sizeof(int), cudaMemcpyHostToDevice,
                           (cudaStream_t)stream) == cudaSuccess
               ? FLEX_OK
               : FLEX_ECUDA;
}

int flex_check_status(void* ws, void* stream)
{
    if (!ws || !aligned(ws, 256)) return FLEX_EINVAL;
    cudaStream_t s = (cudaStream_t)stream;
    if (cudaStreamSynchronize(s) != cudaSuccess) return FLEX_ECUDA;
    flex::WsHeader h;
    if (cudaMemcpyAsync(&h, ws, sizeof(h), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return FLEX_ECUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return FLEX_ECUDA;
    if (h.status != FLEX_OK) {
        if (cudaMemsetAsync(ws, 0, sizeof(int), s) != cudaSuccess) return FLEX_ECUDA;
        if (cudaStreamSynchronize(s) != cudaSuccess) return FLEX_ECUDA;
        return h.status;
    }
    return cudaGetLastError() == cudaSuccess ? FLEX_OK : FLEX_ECUDA;
}

}  // extern "C"
