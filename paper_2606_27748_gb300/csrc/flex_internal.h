// Internal declarations shared by the host API and the kernel translation units.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stddef.h>
#include <stdint.h>

#include "flexattn.h"

namespace flex {

// Workspace layout.  The first 256 bytes hold control words; the rest is scratch whose
// meaning depends on the entry point.
struct WsHeader {
    int status;          // FLEX_OK or FLEX_ETIMEOUT, set by kernels, cleared by check
    int timeout_where;   // diagnostic: which wait gave up
    unsigned int ticket; // dynamic work counter of persistent kernels
    int stall_cycles;    // diagnostic (flex_debug_stall): 0, or the limit of a wait that
                         // nothing ends, taken by the causal forward before any work
    unsigned int pad[60];
};
static_assert(sizeof(WsHeader) == 256, "header is 256 bytes");
// Kernels receive &header.status; the stall limit is the fourth int of the header.
constexpr int kStallWord = 3;
static_assert(offsetof(WsHeader, stall_cycles) == kStallWord * sizeof(int), "header layout");

struct Problem {
    int B, H, N, d, M;
    int bf16;       // storage type of activations: 1 = bf16, 0 = fp32
    int nonstat;    // 1 = nonstationary (W2 given)
    int causal;
};

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Adds n to the count of kernels enqueued by the library (flex_kernel_launches).
void add_launches(int n);

// ---- SIMT path (fp32 arithmetic; any supported dtype) --------------------------------
size_t simt_fwd_smem_bytes(const Problem& p, int chunk);
size_t simt_bwd_smem_bytes(const Problem& p, int chunk);
int simt_pick_chunk_fwd(const Problem& p);   // 0 if nothing fits
int simt_pick_chunk_bwd(const Problem& p);
size_t simt_bwd_ws_bytes(const Problem& p);

cudaError_t launch_featmap(const Problem& p, const void* x, const float* W1, const float* W2,
                           void* phi, cudaStream_t s);
// phi times rowscale[row] (rowscale [B*H*N] or NULL)
cudaError_t launch_featmap_scaled(const Problem& p, const void* x, const float* W1,
                                  const float* W2, const float* rowscale, void* phi,
                                  cudaStream_t s);
// tau: per-head norm prefactor (Sec. 3.2) or NULL; dtau with it in the backward.
cudaError_t launch_simt_fwd(const Problem& p, const void* q, const void* k, const void* v,
                            const float* W1, const float* W2, const float* tau, void* out,
                            float* den, cudaStream_t s);
cudaError_t launch_simt_bwd(const Problem& p, const void* q, const void* k, const void* v,
                            const float* W1, const float* W2, const float* tau,
                            const void* out, const float* den, const void* dout, void* dq,
                            void* dk, void* dv, float* dW1, float* dW2, float* dtau,
                            void* scratch, cudaStream_t s);

// Key weights of the norm prefactor (Sec. 3.2), kw [B*H*N] fp32, for the tensor-core
// forwards: exp(|k|^2 exp(-tau_h)).
cudaError_t launch_key_weights(const Problem& p, const void* k, const float* tau, float* kw,
                               cudaStream_t s);

// ---- recurrent decode step (one token per sequence; fp32 state) ----------------------
size_t decode_ws_bytes(const Problem& p);  // phi(q), phi(k) of the step, fp32
cudaError_t launch_decode(const Problem& p, const void* q, const void* k, const void* v,
                          const float* W1, const float* W2, const float* tau, float* S,
                          float* z, void* out, float* den, void* scratch, int* status,
                          cudaStream_t s);

// ---- tensor-core path (bf16 storage, d = 64, M in {64, 128}) ------------------------
bool tc_fwd_supported(const Problem& p);
int tc_fwd_splits(const Problem& p, int sms);  // segments per sequence (1-3)
// kw: key weights of the norm prefactor or NULL.
cudaError_t launch_tc_fwd(const Problem& p, const void* q, const void* k, const void* v,
                          const float* W1, const float* W2, const float* kw, void* out,
                          float* den, int* status, cudaStream_t s);

bool tc_nc_supported(const Problem& p);
int tc_nc_splits(const Problem& p);
size_t tc_nc_ws_bytes(const Problem& p);
cudaError_t launch_tc_nc(const Problem& p, const void* q, const void* k, const void* v,
                         const float* W1, const float* W2, const float* kw, void* out,
                         float* den, void* scratch, int* status, cudaStream_t s);

bool tc_bwd_supported(const Problem& p);
size_t tc_bwd_ws_bytes(const Problem& p);
int tc_bwd_launches(const Problem& p, bool tau);  // kernels enqueued by launch_tc_bwd
cudaError_t launch_tc_bwd(const Problem& p, const void* q, const void* k, const void* v,
                          const float* W1, const float* W2, const float* tau, const void* out,
                          const float* den, const void* dout, void* dq, void* dk, void* dv,
                          float* dW1, float* dW2, float* dtau, void* scratch, int* status,
                          cudaStream_t s);

// ---- feature map on the tensor cores (bf16, d = 64, M in {64, 128}) ------------------
bool tc_featmap_supported(const Problem& p);
cudaError_t launch_tc_featmap(const Problem& p, const void* x, const float* W1, const float* W2,
                              const float* rowscale, void* phi, int* status, cudaStream_t s);

// ---- attention-weight distillation loss (tensor cores: bf16, d = 64, M in {64, 128}) ---
bool tc_awd_supported(const Problem& p);
size_t tc_awd_part_floats(const Problem& p);  // partial slots [B*H][query blocks]
// pq, pk: phi(q) and the key-weighted phi(k), [B*H][N][2M] bf16; loss [B*H] fp32
cudaError_t launch_tc_awd(const Problem& p, const void* q, const void* k, const void* pq,
                          const void* pk, float* part, float* loss, int* status, cudaStream_t s);
// Loss (loss may be NULL) and its gradient with respect to W1, W2, tau, weighted by dloss
// [B*H]: the loss kernel writes per-row statistics rowstat [B*H*N], then the gradient
// kernel fills slots [tc_awd_slot_floats] and dtau_part [2*B*H], reduced into dW1, dW2,
// dtau.  kw: key weights (with tau) or NULL.
size_t tc_awd_slot_floats(const Problem& p);
cudaError_t launch_tc_awd_bwd(const Problem& p, const void* q, const void* k, const void* pq,
                              const void* pk, const float* W1, const float* W2, const float* kw,
                              const float* tau, const float* dloss, float* part, float* loss,
                              float4* rowstat, float* slots, float* dtau_part, float* dW1,
                              float* dW2, float* dtau, int* status, cudaStream_t s);

}  // namespace flex
