/*
 * flexattn.h -- C ABI of the GB300 (sm_103a) random-Fourier-feature linear attention
 * library (Flexformer: learnable spectral frequencies, stationary and nonstationary).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * Tensors (device pointers, contiguous, row-major):
 *   q, k, v, out, dout, dq, dk, dv : [B][H][N][d]   in `dtype` (fp32 or bf16)
 *   phi                            : [B][H][N][2M]  in `dtype`
 *   W1, W2, dW1, dW2               : [H][M][d]      fp32, one frequency set per head
 *   den                            : [B][H][N]      fp32
 * W2 == NULL selects the stationary variant (Flexformer_s, Sec. 3.2); a non-NULL W2 selects
 * the nonstationary variant (Flexformer_n, Eq. phi_non) with frequency pairs (W1, W2).
 * The feature dimension is d' = 2M (Appendix "Complexity Analysis").
 *
 * Feature map (scale sigma = 1, i.e. M^{-1/2} for both variants):
 *   stationary    phi(x) = M^{-1/2} [cos(W1 x), sin(W1 x)]                     (Eq. phi_n)
 *   nonstationary u = (W1+W2)/2 x,  w = (W1-W2)/2 x,
 *                 phi(x) = M^{-1/2} [cos u * cos w, sin u * cos w]              (Eq. phi_non)
 * all cosine features first, then all sine features.
 *
 * Attention (Eq. linear att):
 *   out_i = phi(q_i)^T S_i / den_i,  den_i = phi(q_i)^T z_i,
 *   S_i = sum_j phi(k_j) v_j^T,  z_i = sum_j phi(k_j),
 * with j <= i when causal (the diagonal is included) and all j otherwise.  The
 * denominator is used as computed: no epsilon, no clamp.
 *
 * Ownership and ordering: the caller owns every buffer.  The library never allocates,
 * frees or synchronises (except flex_check_status); all work is enqueued on `stream`
 * (a cudaStream_t; NULL means the legacy default stream) of the current device.
 * Scratch memory is the caller's workspace `ws` of at least flex_workspace_bytes()
 * bytes, 256-byte aligned and zero-filled before its first use (kernels leave its
 * control words as they found them); one workspace must not be used by two calls that
 * may run concurrently.
 *
 * Errors: every entry point returns FLEX_OK or a negative flex_status and enqueues
 * nothing on error.  Kernels that give up on the device (a bounded wait that ran out)
 * record FLEX_ETIMEOUT in the workspace; flex_check_status() reports it.
 */
#ifndef FLEXATTN_H
#define FLEXATTN_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { FLEX_F32 = 0, FLEX_BF16 = 1 } flex_dtype;

typedef struct {
    int B;      /* batch */
    int H;      /* heads */
    int N;      /* sequence length, >= 1 */
    int d;      /* head size */
    int M;      /* frequencies per set; features d' = 2M */
    int dtype;  /* flex_dtype of q, k, v, out, phi, dout, dq, dk, dv */
} flex_shape;

enum flex_status {
    FLEX_OK = 0,
    FLEX_EINVAL = -1,       /* NULL or misaligned pointer, N < 1, W2/dW2 mismatch, ... */
    FLEX_EUNSUPPORTED = -2, /* valid but unsupported shape/dtype combination */
    FLEX_EWORKSPACE = -3,   /* ws_bytes smaller than flex_workspace_bytes() */
    FLEX_ECUDA = -4,        /* a CUDA launch or runtime call failed */
    FLEX_ETIMEOUT = -5      /* a device-side bounded wait gave up (see flex_check_status) */
};

/* Human-readable text for a flex_status value. */
const char* flex_strerror(int status);

/* Workspace bytes needed by flex_linattn_fwd (backward = 0) or flex_linattn_bwd
 * (backward = 1) for this shape; 0 if the shape is invalid or unsupported. */
size_t flex_workspace_bytes(const flex_shape* shape, int causal, int backward);

/* Feature map phi of Eq. phi_n (W2 == NULL) or Eq. phi_non (W2 != NULL), written out.
 * x: [B][H][N][d], phi: [B][H][N][2M], both in shape->dtype, scaled by M^{-1/2}.  bf16
 * with d = 64 and M in {64, 128} projects on the tensor cores (frequencies rounded to
 * bf16); other shapes use fp32 CUDA-core arithmetic.  This and flex_awd_loss are the only
 * entry points that write phi to memory; the attention entry points keep it on chip. */
int flex_featmap(const flex_shape* shape, const void* x, const float* W1, const float* W2,
                 void* phi, void* stream);

/* Forward linear attention, Eq. (linear att) with the feature map above.
 * tau: NULL, or [H] fp32: the norm prefactor of Sec. 3.2, phi~(x) = exp(|x|^2 / exp(tau_h))
 * phi(x) on queries and keys.  The query's factor cancels in every row, so only the key
 * weight w_j = exp(|k_j|^2 exp(-tau_h)) is applied (to k_j's share of both sums); the
 * weight overflows fp32 when |k_j|^2 exp(-tau_h) > 88.
 * out: [B][H][N][d] in shape->dtype.  den: NULL, or [B][H][N] fp32 receiving
 * den_i = phi(q_i)^T sum_j w_j phi(k_j) (w_j = 1 without tau; the query's factor is not
 * included), needed by flex_linattn_bwd.  ws: workspace of ws_bytes bytes. */
int flex_linattn_fwd(const flex_shape* shape, const void* q, const void* k, const void* v,
                     const float* W1, const float* W2, const float* tau, int causal,
                     void* out, float* den, void* ws, size_t ws_bytes, void* stream);

/* Backward of flex_linattn_fwd: gradients of L = sum(dout * out) with respect to q, k,
 * v and the frequencies.  out and den are the forward's outputs for the same inputs.
 * dq, dk, dv: [B][H][N][d] in shape->dtype.  dW1 (and dW2, which must be NULL exactly
 * when W2 is) are fp32 [H][M][d], summed over the batch and the sequence, overwritten.
 * The paper gives no backward formulas; this is the analytic gradient of Eq. (linear
 * att): with g_i = dout_i / den_i and c_i = -(dout_i . out_i) / den_i,
 *   dphi(q_i) = S_i g_i + c_i z_i,  dphi(k_j) = R_j v_j + r_j,  dv_j = R_j^T phi(k_j),
 *   R_j = sum_{i >= j} phi(q_i) g_i^T,  r_j = sum_{i >= j} c_i phi(q_i)
 * (totals when non-causal), then through the feature map by the chain rule; for the
 * nonstationary variant dW1 = (dU + dV)/2 and dW2 = (dU - dV)/2.  With tau (dtau [H]
 * fp32, NULL exactly when tau is): the formulas hold for the weighted key features
 * w_j phi(k_j); dv_j is multiplied by w_j, and with s_j = phi(k_j) . dphi(k_j) (the
 * gradient with respect to the unweighted features) dk_j gains 2 exp(-tau) s_j k_j and
 * dtau_h = -sum exp(-tau_h) |k_j|^2 s_j over the batch and the sequence (overwritten). */
int flex_linattn_bwd(const flex_shape* shape, const void* q, const void* k, const void* v,
                     const float* W1, const float* W2, const float* tau, int causal,
                     const void* out, const float* den, const void* dout, void* dq,
                     void* dk, void* dv, float* dW1, float* dW2, float* dtau, void* ws,
                     size_t ws_bytes, void* stream);

/* flex_linattn_bwd without a workspace, for callers that cannot allocate device memory:
 * for example a host framework whose memory pool owns all of the device's memory and
 * passes its operators only input and output pointers, or a latency-critical path that
 * must not call cudaMalloc/cudaFree, which can synchronise the device.  (The paper has
 * no counterpart; this is a convenience of this library.)
 * Same arguments, layouts and results as flex_linattn_bwd without the norm prefactor,
 * minus tau, dtau, ws and ws_bytes.  It always runs the fp32 CUDA-core backward (two
 * kernels), never the tensor-core one, so for bf16 storage its results agree with
 * flex_linattn_bwd's within the bf16 tolerance rather than bit for bit, and its speed
 * differs.  The scratch is one array of 4 MiB (2^20 floats) in the library's own device
 * memory, which every GPU that loads the library keeps until the process exits; it must
 * hold B * H * (Mc * d + 1) floats (Mc = M, or 2M when W2 is given), else FLEX_EWORKSPACE
 * is returned and nothing runs.  Nothing is allocated or freed.  All calls on a device
 * share that array and it keeps the last call's contents, so two calls whose work may
 * overlap on the GPU (different streams, or different host threads) race and must be
 * ordered by the caller.  The first call on a device (and the first after its context
 * was replaced, e.g. by cudaDeviceReset) looks the array's address up with that device
 * current; make that first call before any stream capture. */
int flex_linattn_bwd_noalloc(const flex_shape* shape, const void* q, const void* k,
                             const void* v, const float* W1, const float* W2, int causal,
                             const void* out, const float* den, const void* dout, void* dq,
                             void* dk, void* dv, float* dW1, float* dW2, void* stream);

/* Workspace bytes needed by flex_linattn_decode for this shape (shape->N must be 1); 0 if
 * the shape is invalid. */
size_t flex_decode_workspace_bytes(const flex_shape* shape);

/* One recurrent decode step of the causal form of Eq. (linear att) (the running sums of
 * Sec. 2.2): for each (b, h) the new token's q, k, v ([B][H][d] in shape->dtype;
 * shape->N must be 1) update S += phi(k) v^T and z += phi(k), then
 * out = phi(q)^T S / den with den = phi(q)^T z -- the new token included (j <= i).
 * S: [B][H][2M][d] fp32 and z: [B][H][2M] fp32, caller-owned, read and written in place
 * (zero-filled before a sequence's first token); phi is scaled by M^{-1/2} as in Eq. phi_n
 * / phi_non, so S and z are exactly the paper's running sums.  out: [B][H][d] in
 * shape->dtype; den: NULL or [B][H] fp32.  Stepping through a sequence reproduces
 * flex_linattn_fwd(causal = 1) row by row (with the same tau: the new key's features
 * enter S and z with its weight w).  ws: workspace of at least
 * flex_decode_workspace_bytes() bytes (it holds the step's phi(q), phi(k); a serving loop
 * allocates it once).  Two kernels per call.  Errors: FLEX_EINVAL for NULL or misaligned
 * pointers or N != 1, FLEX_EWORKSPACE, FLEX_EUNSUPPORTED as for the other entry points. */
int flex_linattn_decode(const flex_shape* shape, const void* q, const void* k, const void* v,
                        const float* W1, const float* W2, const float* tau, float* S,
                        float* z, void* out, float* den, void* ws, size_t ws_bytes,
                        void* stream);

/* Workspace bytes needed by flex_awd_loss for this shape; 0 if the shape is invalid or
 * unsupported. */
size_t flex_awd_workspace_bytes(const flex_shape* shape);

/* Attention-weight distillation loss (the loss of the paper's softmax-recovery
 * experiments, appendix "Attention Distillation Setting"): for every (b, h) sequence
 *   loss[b][h] = -(1/N) sum_i sum_j P_ij log R_ij,
 *   P_ij = softmax_j(q_i . k_j / sqrt(d))               (the teacher: softmax attention),
 *   R_ij = A~_ij / sum_l A~_il,  A~_ij = phi~(q_i) . phi~(k_j)   (this kernel's weights),
 * j over all keys, or j <= i when causal; phi~ is the feature map above with the optional
 * norm prefactor tau ([H] fp32 or NULL).  An entry whose R_ij is not positive (random
 * Fourier estimates and row sums can be negative) counts log(1e-6).  Computed blockwise
 * (128 x 128 tiles of scores and kernel values on the tensor cores, online softmax), never
 * materialising the N x N matrices.  q, k: [B][H][N][d] bf16 (d = 64, M in {64, 128});
 * loss: [B][H] fp32, overwritten.  ws: workspace of flex_awd_workspace_bytes() bytes
 * (it holds phi(q) and the key-weighted phi(k), written by a tensor-core feature pass).
 * Launches 4 kernels (5 with tau).  Errors: FLEX_EINVAL for NULL or misaligned pointers,
 * FLEX_EUNSUPPORTED for other shapes or fp32 storage, FLEX_EWORKSPACE. */
int flex_awd_loss(const flex_shape* shape, const void* q, const void* k, const float* W1,
                  const float* W2, const float* tau, int causal, float* loss, void* ws,
                  size_t ws_bytes, void* stream);

/* Workspace bytes needed by flex_awd_loss_bwd for this shape; 0 if the shape is invalid
 * or unsupported. */
size_t flex_awd_bwd_workspace_bytes(const flex_shape* shape);

/* One distillation step's loss and gradient.  The distillation trains only the kernel's
 * parameters (appendix "Attention Distillation Setting": the Transformer is frozen), so
 * the gradient of sum_{b,h} dloss[b][h] loss[b][h] (loss as in flex_awd_loss) is taken
 * with respect to W1, W2 and tau, not q and k.  An entry with R_ij <= 0 is constant
 * (log 1e-6) and has no gradient; on an entry with R_ij > 0,
 *   d loss / d A~_ij = -(1/N) (P_ij / A~_ij - c_i / D_i),
 * c_i the teacher mass on row i's entries with R_ij > 0 and D_i the row sum.  Near
 * A~_ij = 0 the first term has a pole, so where some estimates are negative the gradient
 * is ill-conditioned; the computation is meant for inputs whose weights are positive.
 * q, k: [B][H][N][d] bf16 (d = 64, M in {64, 128}); dloss: [B][H] fp32 (device);
 * loss: NULL or [B][H] fp32, overwritten; dW1, dW2: [H][M][d] fp32, overwritten (dW2 given
 * exactly when W2 is); dtau: [H] fp32, overwritten (given exactly when tau is).
 * ws: workspace of flex_awd_bwd_workspace_bytes() bytes.  Launches 6 kernels (5 without
 * loss, one more with tau): the feature passes, the loss kernel (which also records each
 * row's softmax normaliser, row-sum sign and c_i / D_i), its reduction, one gradient kernel
 * (a query side and a key side, blockwise on the tensor cores; the chain rule through the
 * feature map runs in the same kernel) and a fixed-order reduction, so the result does not
 * depend on scheduling.  Errors as for flex_awd_loss, and FLEX_EINVAL when dW2 or dtau is
 * given without W2 or tau (or missing with it). */
int flex_awd_loss_bwd(const flex_shape* shape, const void* q, const void* k, const float* W1,
                      const float* W2, const float* tau, int causal, const float* dloss,
                      float* loss, float* dW1, float* dW2, float* dtau, void* ws,
                      size_t ws_bytes, void* stream);

/* Cumulative number of kernels this library has enqueued in this process (all entry
 * points, all devices).  Lets a caller count the launches inside a timed region. */
unsigned long long flex_kernel_launches(void);

/* Synchronises `stream`, then returns FLEX_ETIMEOUT if a kernel that used `ws` gave up
 * on a bounded wait since the workspace was last checked, FLEX_ECUDA on a pending CUDA
 * error, else FLEX_OK.  Clears the recorded status. */
int flex_check_status(void* ws, void* stream);

/* Diagnostic of the bounded waits (the paper has no counterpart).  Enqueues on `stream`
 * a write of `cycles` into the header of workspace `ws` (ws_bytes >= 256).  While it is
 * nonzero, every CTA of the causal tensor-core forward (flex_linattn_fwd with causal = 1,
 * bf16, d = 64, M in {64, 128}) first waits at most `cycles` clocks, during its set-up and
 * before it issues any copy or tensor-core operation, on an mbarrier that nothing arrives
 * on; the wait runs out as a wait for a lost arrival would (FLEX_ETIMEOUT recorded in
 * `ws`, reported by flex_check_status), the CTA frees its tensor memory and exits, and
 * `out`/`den` are left unwritten.  flex_debug_stall(ws, ws_bytes, 0, stream) restores
 * normal operation.  Other entry points ignore the value.  Errors: FLEX_EINVAL (NULL or
 * misaligned ws, cycles < 0), FLEX_EWORKSPACE, FLEX_ECUDA. */
int flex_debug_stall(void* ws, size_t ws_bytes, int cycles, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* FLEXATTN_H */
