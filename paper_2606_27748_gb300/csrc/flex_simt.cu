// SIMT kernels: fp32 arithmetic on the CUDA cores, one CTA per (b, h) sequence.
//
// These kernels serve the fp32 storage type, whose tolerance (relative L2 <= 1e-4)
// excludes bf16/tf32 tensor-core operands, and the feature-map entry point.  They run the
// chunked form of Eq. (linear att): inside a chunk of C tokens the masked C x C kernel
// matrix phi(Q) phi(K)^T is applied directly, across chunks the running state
// S = sum phi(k) v^T and z = sum phi(k) carries the prefix.  z rides in S as column d
// (v is extended with a constant 1), so numerator and denominator share every product.
//
// Inside the attention kernels the features are unscaled, phi' = [cos, sin] (times cos w
// for the nonstationary map): the global factor M^{-1/2} of Eq. phi_n / phi_non cancels in
// out and in every gradient, and only the stored denominator is rescaled, den = den'/M.
//
// Norm prefactor (Sec. 3.2, optional, tau per head): phi~(x) = exp(|x|^2 / exp(tau)) phi(x).
// The query's factor cancels row by row; the key's is a weight w_j, carried by turning the
// key rows [v_j | 1] into [w_j v_j | w_j].  The backward then multiplies dv_j by w_j and,
// with s_j = phi(k_j) . dphi(k_j), adds 2 exp(-tau) s_j k_j to dk_j and
// -exp(-tau) |k_j|^2 s_j to dtau.
#include "flex_internal.h"

#include <math.h>

#include <algorithm>

namespace flex {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxDwPerThread = 64;  // Mc * d <= kThreads * 64

__device__ __forceinline__ float load_act(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float load_act(const __nv_bfloat16* p, size_t i)
{
    return __bfloat162float(p[i]);
}
__device__ __forceinline__ void store_act(float* p, size_t i, float x) { p[i] = x; }
__device__ __forceinline__ void store_act(__nv_bfloat16* p, size_t i, float x)
{
    p[i] = __float2bfloat16_rn(x);
}

// Projection rows of one head into shared memory, row stride d + 1:
// stationary: W1 (M rows); nonstationary: U = (W1+W2)/2 then V = (W1-W2)/2 (2M rows).
__device__ void load_projection(const Problem& p, const float* W1, const float* W2, int h,
                                float* W)
{
    const int d = p.d, M = p.M;
    const float* w1 = W1 + (size_t)h * M * d;
    const float* w2 = p.nonstat ? W2 + (size_t)h * M * d : nullptr;
    for (int idx = threadIdx.x; idx < M * d; idx += blockDim.x) {
        int m = idx / d, i = idx % d;
        if (!p.nonstat) {
            W[m * (d + 1) + i] = w1[idx];
        } else {
            W[m * (d + 1) + i] = 0.5f * (w1[idx] + w2[idx]);
            W[(M + m) * (d + 1) + i] = 0.5f * (w1[idx] - w2[idx]);
        }
    }
}

template <typename T>
__device__ void load_rows(const T* src, size_t base, int rows, int d, float* dst, int stride)
{
    for (int idx = threadIdx.x; idx < rows * d; idx += blockDim.x) {
        int t = idx / d, i = idx % d;
        dst[t * stride + i] = load_act(src, base + (size_t)t * d + i);
    }
}

// Unscaled features of `rows` vectors X[t][0..d) into P[t][0..2M), row stride pstride.
__device__ void features(const Problem& p, const float* X, int rows, const float* W, float* P,
                         int pstride)
{
    const int d = p.d, M = p.M;
    for (int idx = threadIdx.x; idx < rows * M; idx += blockDim.x) {
        int t = idx / M, m = idx % M;
        const float* x = X + t * d;
        const float* wa = W + m * (d + 1);
        float a = 0.f;
        for (int i = 0; i < d; ++i) a = fmaf(x[i], wa[i], a);
        float sa, ca;
        sincosf(a, &sa, &ca);
        if (!p.nonstat) {
            P[t * pstride + m] = ca;
            P[t * pstride + M + m] = sa;
        } else {
            const float* wb = W + (M + m) * (d + 1);
            float w = 0.f;
            for (int i = 0; i < d; ++i) w = fmaf(x[i], wb[i], w);
            float cw = cosf(w);
            P[t * pstride + m] = ca * cw;
            P[t * pstride + M + m] = sa * cw;
        }
    }
}

// ------------------------------------------------------------------------------------
// Feature map entry point (writes phi, scaled by M^{-1/2}).
// ------------------------------------------------------------------------------------
template <typename T>
__global__ void featmap_kernel(Problem p, const T* x, const float* W1, const float* W2, T* phi,
                               float scale, const float* rowscale)
{
    const int d = p.d, M = p.M;
    const size_t rows = (size_t)p.B * p.H * p.N;
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < rows * M;
         idx += (size_t)gridDim.x * blockDim.x) {
        size_t row = idx / M;
        int m = (int)(idx % M);
        int h = (int)((row / p.N) % p.H);
        const float* w1 = W1 + ((size_t)h * M + m) * d;
        float a = 0.f, w = 0.f;
        if (!p.nonstat) {
            for (int i = 0; i < d; ++i) a = fmaf(load_act(x, row * d + i), w1[i], a);
        } else {
            const float* w2 = W2 + ((size_t)h * M + m) * d;
            for (int i = 0; i < d; ++i) {
                float xi = load_act(x, row * d + i);
                a = fmaf(xi, 0.5f * (w1[i] + w2[i]), a);
                w = fmaf(xi, 0.5f * (w1[i] - w2[i]), w);
            }
        }
        float sa, ca;
        sincosf(a, &sa, &ca);
        float cw = (p.nonstat ? cosf(w) : 1.f) * scale * (rowscale ? rowscale[row] : 1.f);
        store_act(phi, row * 2 * M + m, ca * cw);
        store_act(phi, row * 2 * M + M + m, sa * cw);
    }
}

// ------------------------------------------------------------------------------------
// Forward.
// ------------------------------------------------------------------------------------
// [v_j | 1] -> [w_j v_j | w_j] for the key rows of a chunk, w_j = exp(|k_j|^2 itau).
__device__ void weight_keys(const float* Xk, int rows, int d, float itau, float* Vx)
{
    for (int j = threadIdx.x; j < rows; j += blockDim.x) {
        float n2 = 0.f;
        for (int e = 0; e < d; ++e) n2 = fmaf(Xk[j * d + e], Xk[j * d + e], n2);
        const float w = expf(n2 * itau);
        for (int e = 0; e < d; ++e) Vx[j * (d + 1) + e] *= w;
        Vx[j * (d + 1) + d] = w;
    }
}

struct FwdLayout {
    size_t W, S, Xq, Xk, Vx, Pq, Pk, A, O, total;  // offsets in floats
};

__host__ __device__ inline FwdLayout fwd_layout(const Problem& p, int C)
{
    const int d = p.d, D = 2 * p.M, Mc = p.nonstat ? 2 * p.M : p.M;
    FwdLayout L;
    size_t o = 0;
    L.W = o;  o += (size_t)Mc * (d + 1);
    L.S = o;  o += (size_t)D * (d + 1);
    L.Xq = o; o += (size_t)C * d;
    L.Xk = o; o += (size_t)C * d;
    L.Vx = o; o += (size_t)C * (d + 1);
    L.Pq = o; o += (size_t)C * (D + 1);
    L.Pk = o; o += (size_t)C * (D + 1);
    L.A = o;  o += (size_t)C * C;
    L.O = o;  o += (size_t)C * (d + 1);
    L.total = o;
    return L;
}

// S[f][e] += sum_{j < rows} Pk[j][f] * Vx[j][e]
__device__ void state_update(const float* Pk, const float* Vx, int rows, int D, int d,
                             float* S)
{
    for (int idx = threadIdx.x; idx < D * (d + 1); idx += blockDim.x) {
        int f = idx / (d + 1), e = idx % (d + 1);
        float acc = S[idx];
        for (int j = 0; j < rows; ++j) acc = fmaf(Pk[j * (D + 1) + f], Vx[j * (d + 1) + e], acc);
        S[idx] = acc;
    }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) simt_fwd_kernel(Problem p, int C, const T* q,
                                                            const T* k, const T* v,
                                                            const float* W1, const float* W2,
                                                            const float* tau, T* out,
                                                            float* den)
{
    extern __shared__ float sm[];
    const int d = p.d, D = 2 * p.M, N = p.N;
    const int bh = blockIdx.x, h = bh % p.H;
    const size_t base = (size_t)bh * N * d;
    const FwdLayout L = fwd_layout(p, C);
    float *W = sm + L.W, *S = sm + L.S, *Xq = sm + L.Xq, *Xk = sm + L.Xk, *Vx = sm + L.Vx;
    float *Pq = sm + L.Pq, *Pk = sm + L.Pk, *A = sm + L.A, *O = sm + L.O;
    const float inv_m = 1.0f / (float)p.M;
    const float itau = tau ? expf(-tau[h]) : 0.f;

    load_projection(p, W1, W2, h, W);
    for (int idx = threadIdx.x; idx < D * (d + 1); idx += blockDim.x) S[idx] = 0.f;
    for (int idx = threadIdx.x; idx < C; idx += blockDim.x) Vx[idx * (d + 1) + d] = 1.f;
    __syncthreads();

    if (!p.causal) {  // totals S, z over the whole sequence first
        for (int t0 = 0; t0 < N; t0 += C) {
            const int CL = min(C, N - t0);
            load_rows(k, base + (size_t)t0 * d, CL, d, Xk, d);
            load_rows(v, base + (size_t)t0 * d, CL, d, Vx, d + 1);
            __syncthreads();
            if (tau) weight_keys(Xk, CL, d, itau, Vx);
            features(p, Xk, CL, W, Pk, D + 1);
            __syncthreads();
            state_update(Pk, Vx, CL, D, d, S);
            __syncthreads();
        }
    }
    for (int t0 = 0; t0 < N; t0 += C) {
        const int CL = min(C, N - t0);
        load_rows(q, base + (size_t)t0 * d, CL, d, Xq, d);
        if (p.causal) {
            load_rows(k, base + (size_t)t0 * d, CL, d, Xk, d);
            load_rows(v, base + (size_t)t0 * d, CL, d, Vx, d + 1);
        }
        __syncthreads();
        if (tau && p.causal) weight_keys(Xk, CL, d, itau, Vx);
        features(p, Xq, CL, W, Pq, D + 1);
        if (p.causal) features(p, Xk, CL, W, Pk, D + 1);
        __syncthreads();
        if (p.causal) {
            for (int idx = threadIdx.x; idx < CL * CL; idx += blockDim.x) {
                int i = idx / CL, j = idx % CL;
                float a = 0.f;
                if (j <= i)
                    for (int f = 0; f < D; ++f) a = fmaf(Pq[i * (D + 1) + f], Pk[j * (D + 1) + f], a);
                A[i * C + j] = a;
            }
            __syncthreads();
        }
        // numerator (columns < d) and denominator (column d) of every row of the chunk
        for (int idx = threadIdx.x; idx < CL * (d + 1); idx += blockDim.x) {
            int i = idx / (d + 1), e = idx % (d + 1);
            float acc = 0.f;
            if (p.causal)
                for (int j = 0; j <= i; ++j) acc = fmaf(A[i * C + j], Vx[j * (d + 1) + e], acc);
            for (int f = 0; f < D; ++f) acc = fmaf(Pq[i * (D + 1) + f], S[f * (d + 1) + e], acc);
            O[i * (d + 1) + e] = acc;
        }
        __syncthreads();
        for (int idx = threadIdx.x; idx < CL * d; idx += blockDim.x) {
            int i = idx / d, e = idx % d;
            store_act(out, base + (size_t)(t0 + i) * d + e, O[i * (d + 1) + e] / O[i * (d + 1) + d]);
        }
        if (den)
            for (int i = threadIdx.x; i < CL; i += blockDim.x)
                den[(size_t)bh * N + t0 + i] = O[i * (d + 1) + d] * inv_m;
        if (p.causal) state_update(Pk, Vx, CL, D, d, S);
        __syncthreads();
    }
}

// ------------------------------------------------------------------------------------
// Backward.
// ------------------------------------------------------------------------------------
struct BwdLayout {
    size_t W, S, Xq, Xk, Vx, Gx, Pq, Pk, dP, A, dA, dAct, Kc, total;
};

__host__ __device__ inline BwdLayout bwd_layout(const Problem& p, int C)
{
    const int d = p.d, D = 2 * p.M, Mc = p.nonstat ? 2 * p.M : p.M;
    BwdLayout L;
    size_t o = 0;
    L.W = o;    o += (size_t)Mc * (d + 1);
    L.S = o;    o += (size_t)D * (d + 1);
    L.Xq = o;   o += (size_t)C * d;
    L.Xk = o;   o += (size_t)C * d;
    L.Vx = o;   o += (size_t)C * (d + 1);
    L.Gx = o;   o += (size_t)C * (d + 1);
    L.Pq = o;   o += (size_t)C * (D + 1);
    L.Pk = o;   o += (size_t)C * (D + 1);
    L.dP = o;   o += (size_t)C * (D + 1);
    L.A = o;    o += (size_t)C * C;
    L.dA = o;   o += (size_t)C * C;
    L.dAct = o; o += (size_t)C * (Mc + 1);
    L.Kc = o;   o += (size_t)C;
    L.total = o;
    return L;
}

// Gx[t] = [dout_t / den'_t, -(dout_t . out_t) / den'_t] with den' = M * den.
template <typename T>
__device__ void load_upstream(const Problem& p, const T* dout, const T* out, const float* den,
                              size_t base, size_t den_base, int rows, float* Gx)
{
    const int d = p.d;
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32, nwarps = blockDim.x / 32;
    for (int t = warp; t < rows; t += nwarps) {
        const float dn = den[den_base + t] * (float)p.M;
        float s = 0.f;
        for (int e = lane; e < d; e += 32) {
            float g = load_act(dout, base + (size_t)t * d + e);
            s = fmaf(g, load_act(out, base + (size_t)t * d + e), s);
            Gx[t * (d + 1) + e] = g / dn;
        }
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
        if (lane == 0) Gx[t * (d + 1) + d] = -s / dn;
    }
}

// Chain rule through the feature map: dAct[t][m] = d/da (stationary) or (du, dw).
__device__ void feature_backward(const Problem& p, const float* X, const float* P,
                                 const float* dP, int rows, const float* W, float* dAct)
{
    const int d = p.d, M = p.M, D = 2 * M, Mc = p.nonstat ? 2 * M : M;
    for (int idx = threadIdx.x; idx < rows * M; idx += blockDim.x) {
        int t = idx / M, m = idx % M;
        const float dc = dP[t * (D + 1) + m], ds = dP[t * (D + 1) + M + m];
        if (!p.nonstat) {
            const float c = P[t * (D + 1) + m], s = P[t * (D + 1) + M + m];
            dAct[t * (Mc + 1) + m] = -s * dc + c * ds;
        } else {
            const float* x = X + t * d;
            const float *wa = W + m * (d + 1), *wb = W + (M + m) * (d + 1);
            float u = 0.f, w = 0.f;
            for (int i = 0; i < d; ++i) {
                u = fmaf(x[i], wa[i], u);
                w = fmaf(x[i], wb[i], w);
            }
            float su, cu, sw, cw;
            sincosf(u, &su, &cu);
            sincosf(w, &sw, &cw);
            dAct[t * (Mc + 1) + m] = cw * (-su * dc + cu * ds);
            dAct[t * (Mc + 1) + M + m] = -sw * (cu * dc + su * ds);
        }
    }
}

// dx[t][i] = sum_m dAct[t][m] W[m][i] (+ xcoef[t] X[t][i], the key prefactor's term);
// dW[m][i] += sum_t dAct[t][m] X[t][i].
template <typename T>
__device__ void project_back(const Problem& p, const float* X, const float* dAct, int rows,
                             const float* W, T* dx, size_t base, float* dw_acc,
                             const float* xcoef)
{
    const int d = p.d, Mc = p.nonstat ? 2 * p.M : p.M;
    for (int idx = threadIdx.x; idx < rows * d; idx += blockDim.x) {
        int t = idx / d, i = idx % d;
        float acc = 0.f;
        for (int m = 0; m < Mc; ++m) acc = fmaf(dAct[t * (Mc + 1) + m], W[m * (d + 1) + i], acc);
        if (xcoef) acc = fmaf(xcoef[t], X[t * d + i], acc);
        store_act(dx, base + (size_t)t * d + i, acc);
    }
#pragma unroll
    for (int r = 0; r < kMaxDwPerThread; ++r) {
        int e = r * kThreads + threadIdx.x;
        if (e < Mc * d) {
            int m = e / d, i = e % d;
            float acc = dw_acc[r];
            for (int t = 0; t < rows; ++t) acc = fmaf(dAct[t * (Mc + 1) + m], X[t * d + i], acc);
            dw_acc[r] = acc;
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(kThreads) simt_bwd_kernel(
    Problem p, int C, const T* q, const T* k, const T* v, const float* W1, const float* W2,
    const float* tau, const T* out, const float* den, const T* dout, T* dq, T* dk, T* dv,
    float* dw_part, float* dtau_part)
{
    extern __shared__ float sm[];
    const int d = p.d, D = 2 * p.M, N = p.N, Mc = p.nonstat ? 2 * p.M : p.M;
    const int bh = blockIdx.x, h = bh % p.H;
    const size_t base = (size_t)bh * N * d, den_base = (size_t)bh * N;
    const BwdLayout L = bwd_layout(p, C);
    float *W = sm + L.W, *S = sm + L.S, *Xq = sm + L.Xq, *Xk = sm + L.Xk, *Vx = sm + L.Vx;
    float *Gx = sm + L.Gx, *Pq = sm + L.Pq, *Pk = sm + L.Pk, *dP = sm + L.dP;
    float *A = sm + L.A, *dA = sm + L.dA, *dAct = sm + L.dAct, *Kc = sm + L.Kc;
    const float itau = tau ? expf(-tau[h]) : 0.f;
    float dtau_acc = 0.f;
    // |k_0|^2 of the sequence: dtau = -exp(-tau) sum_j (|k_j|^2 - |k_0|^2) s_j (the s_j of a
    // sequence sum to zero, as every output row is invariant to a common key-weight scale)
    float n20 = 0.f;
    if (tau)
        for (int e = 0; e < d; ++e) {
            const float x = load_act(k, base + e);
            n20 = fmaf(x, x, n20);
        }

    float dw_acc[kMaxDwPerThread];
#pragma unroll
    for (int r = 0; r < kMaxDwPerThread; ++r) dw_acc[r] = 0.f;

    load_projection(p, W1, W2, h, W);
    for (int idx = threadIdx.x; idx < D * (d + 1); idx += blockDim.x) S[idx] = 0.f;
    for (int idx = threadIdx.x; idx < C; idx += blockDim.x) Vx[idx * (d + 1) + d] = 1.f;
    __syncthreads();

    // ---- dq: forward direction with S_i, z_i ----
    if (!p.causal) {
        for (int t0 = 0; t0 < N; t0 += C) {
            const int CL = min(C, N - t0);
            load_rows(k, base + (size_t)t0 * d, CL, d, Xk, d);
            load_rows(v, base + (size_t)t0 * d, CL, d, Vx, d + 1);
            __syncthreads();
            if (tau) weight_keys(Xk, CL, d, itau, Vx);
            features(p, Xk, CL, W, Pk, D + 1);
            __syncthreads();
            state_update(Pk, Vx, CL, D, d, S);
            __syncthreads();
        }
    }
    for (int t0 = 0; t0 < N; t0 += C) {
        const int CL = min(C, N - t0);
        const size_t off = base + (size_t)t0 * d;
        load_rows(q, off, CL, d, Xq, d);
        load_upstream(p, dout, out, den, off, den_base + t0, CL, Gx);
        if (p.causal) {
            load_rows(k, off, CL, d, Xk, d);
            load_rows(v, off, CL, d, Vx, d + 1);
        }
        __syncthreads();
        if (tau && p.causal) {
            weight_keys(Xk, CL, d, itau, Vx);
            __syncthreads();
        }
        features(p, Xq, CL, W, Pq, D + 1);
        if (p.causal) features(p, Xk, CL, W, Pk, D + 1);
        if (p.causal)
            for (int idx = threadIdx.x; idx < CL * CL; idx += blockDim.x) {
                int i = idx / CL, j = idx % CL;
                float a = 0.f;
                if (j <= i)
                    for (int e = 0; e <= d; ++e) a = fmaf(Gx[i * (d + 1) + e], Vx[j * (d + 1) + e], a);
                dA[i * C + j] = a;
            }
        __syncthreads();
        for (int idx = threadIdx.x; idx < CL * D; idx += blockDim.x) {
            int i = idx / D, f = idx % D;
            float acc = 0.f;
            if (p.causal)
                for (int j = 0; j <= i; ++j) acc = fmaf(dA[i * C + j], Pk[j * (D + 1) + f], acc);
            for (int e = 0; e <= d; ++e) acc = fmaf(S[f * (d + 1) + e], Gx[i * (d + 1) + e], acc);
            dP[i * (D + 1) + f] = acc;
        }
        __syncthreads();
        if (p.causal) state_update(Pk, Vx, CL, D, d, S);
        feature_backward(p, Xq, Pq, dP, CL, W, dAct);
        __syncthreads();
        project_back(p, Xq, dAct, CL, W, dq, off, dw_acc, nullptr);
        __syncthreads();
    }

    // ---- dk, dv: reverse direction with R_j, r_j (S's buffer is reused for R) ----
    for (int idx = threadIdx.x; idx < D * (d + 1); idx += blockDim.x) S[idx] = 0.f;
    __syncthreads();
    float* R = S;
    if (!p.causal) {
        for (int t0 = 0; t0 < N; t0 += C) {
            const int CL = min(C, N - t0);
            const size_t off = base + (size_t)t0 * d;
            load_rows(q, off, CL, d, Xq, d);
            load_upstream(p, dout, out, den, off, den_base + t0, CL, Gx);
            __syncthreads();
            features(p, Xq, CL, W, Pq, D + 1);
            __syncthreads();
            state_update(Pq, Gx, CL, D, d, R);
            __syncthreads();
        }
    }
    const int nchunks = (N + C - 1) / C;
    for (int c = nchunks - 1; c >= 0; --c) {
        const int t0 = c * C, CL = min(C, N - t0);
        const size_t off = base + (size_t)t0 * d;
        load_rows(k, off, CL, d, Xk, d);
        load_rows(v, off, CL, d, Vx, d + 1);
        if (p.causal) {
            load_rows(q, off, CL, d, Xq, d);
            load_upstream(p, dout, out, den, off, den_base + t0, CL, Gx);
        }
        __syncthreads();
        if (tau) {
            weight_keys(Xk, CL, d, itau, Vx);
            __syncthreads();
        }
        features(p, Xk, CL, W, Pk, D + 1);
        if (p.causal) features(p, Xq, CL, W, Pq, D + 1);
        __syncthreads();
        if (p.causal)
            for (int idx = threadIdx.x; idx < CL * CL; idx += blockDim.x) {
                int i = idx / CL, j = idx % CL;
                float a = 0.f, da = 0.f;
                if (j <= i) {
                    for (int f = 0; f < D; ++f) a = fmaf(Pq[i * (D + 1) + f], Pk[j * (D + 1) + f], a);
                    for (int e = 0; e <= d; ++e) da = fmaf(Gx[i * (d + 1) + e], Vx[j * (d + 1) + e], da);
                }
                A[i * C + j] = a;
                dA[i * C + j] = da;
            }
        __syncthreads();
        for (int idx = threadIdx.x; idx < CL * D; idx += blockDim.x) {
            int j = idx / D, f = idx % D;
            float acc = 0.f;
            if (p.causal)
                for (int i = j; i < CL; ++i) acc = fmaf(dA[i * C + j], Pq[i * (D + 1) + f], acc);
            for (int e = 0; e <= d; ++e) acc = fmaf(R[f * (d + 1) + e], Vx[j * (d + 1) + e], acc);
            dP[j * (D + 1) + f] = acc;
        }
        for (int idx = threadIdx.x; idx < CL * d; idx += blockDim.x) {
            int j = idx / d, e = idx % d;
            float acc = 0.f;
            if (p.causal)
                for (int i = j; i < CL; ++i) acc = fmaf(A[i * C + j], Gx[i * (d + 1) + e], acc);
            for (int f = 0; f < D; ++f) acc = fmaf(R[f * (d + 1) + e], Pk[j * (D + 1) + f], acc);
            if (tau) acc *= Vx[j * (d + 1) + d];  // dv_j = w_j R_j^T phi(k_j)
            store_act(dv, off + (size_t)j * d + e, acc);
        }
        __syncthreads();
        if (tau)  // s_j = phi(k_j) . dphi(k_j): dk_j += 2 itau s_j k_j, dtau -= itau |k_j|^2 s_j
            for (int j = threadIdx.x; j < CL; j += blockDim.x) {
                float sj = 0.f, n2 = 0.f;
                for (int f = 0; f < D; ++f) sj = fmaf(Pk[j * (D + 1) + f], dP[j * (D + 1) + f], sj);
                for (int e = 0; e < d; ++e) n2 = fmaf(Xk[j * d + e], Xk[j * d + e], n2);
                Kc[j] = 2.f * itau * sj;
                dtau_acc = fmaf(-itau * (n2 - n20), sj, dtau_acc);
            }
        if (p.causal) state_update(Pq, Gx, CL, D, d, R);
        feature_backward(p, Xk, Pk, dP, CL, W, dAct);
        __syncthreads();
        project_back(p, Xk, dAct, CL, W, dk, off, dw_acc, tau ? Kc : nullptr);
        __syncthreads();
    }

    float* part = dw_part + (size_t)bh * Mc * d;
#pragma unroll
    for (int r = 0; r < kMaxDwPerThread; ++r) {
        int e = r * kThreads + threadIdx.x;
        if (e < Mc * d) part[e] = dw_acc[r];
    }
    if (tau) {  // this sequence's dtau: warp sums, then the warps in order
        for (int o = 16; o > 0; o >>= 1) dtau_acc += __shfl_xor_sync(0xffffffffu, dtau_acc, o);
        __syncthreads();
        if ((threadIdx.x & 31) == 0) Kc[threadIdx.x >> 5] = dtau_acc;
        __syncthreads();
        if (threadIdx.x == 0) {
            float t = 0.f;
            for (int w = 0; w < kThreads / 32; ++w) t += Kc[w];
            dtau_part[bh] = t;
        }
    }
}

// Key weights of the norm prefactor for the tensor-core forwards: kw[row] =
// exp(|k_row|^2 exp(-tau_h)) for every row of k [B*H*N][d]; one thread per row, vector
// loads of 4 elements (d % 4 == 0).
template <typename T>
__global__ void __launch_bounds__(kThreads) key_weights_kernel(Problem p, const T* k,
                                                               const float* tau, float* kw)
{
    const size_t rows = (size_t)p.B * p.H * p.N;
    for (size_t r = (size_t)blockIdx.x * blockDim.x + threadIdx.x; r < rows;
         r += (size_t)gridDim.x * blockDim.x) {
        const T* x = k + r * p.d;
        float n2 = 0.f;
        for (int e = 0; e < p.d; e += 4) {
            float v[4];
            if constexpr (sizeof(T) == 4) {
                const float4 f = *reinterpret_cast<const float4*>(x + e);
                v[0] = f.x; v[1] = f.y; v[2] = f.z; v[3] = f.w;
            } else {
                const uint2 u = *reinterpret_cast<const uint2*>(x + e);
                v[0] = __uint_as_float(u.x << 16); v[1] = __uint_as_float(u.x & 0xffff0000u);
                v[2] = __uint_as_float(u.y << 16); v[3] = __uint_as_float(u.y & 0xffff0000u);
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) n2 = fmaf(v[i], v[i], n2);
        }
        const int h = (int)((r / p.N) % p.H);
        kw[r] = expf(n2 * expf(-tau[h]));
    }
}

// The same for bf16 rows of d = 64 (the tensor-core shapes): 8 lanes per row, one 16-byte
// load each (fully coalesced), 4 rows in flight per lane, the 8 partial sums combined by
// xor shuffles.
__global__ void __launch_bounds__(kThreads) key_weights_bf16_d64_kernel(Problem p,
                                                                         const __nv_bfloat16* k,
                                                                         const float* tau,
                                                                         float* kw)
{
    constexpr int kUnroll = 4;
    const size_t rows = (size_t)p.B * p.H * p.N;
    const int lane = threadIdx.x & 31, sub = lane & 7;
    const size_t warps = (size_t)gridDim.x * (blockDim.x / 32);
    const size_t gw = (size_t)blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5);
    for (size_t r0 = gw * 4 * kUnroll; r0 < rows; r0 += warps * 4 * kUnroll) {
        uint4 x[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const size_t r = r0 + 4 * u + (lane >> 3);
            x[u] = r < rows ? *reinterpret_cast<const uint4*>(k + r * 64 + 8 * sub)
                            : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
            const uint32_t wv[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
            float n2 = 0.f;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float a = __uint_as_float(wv[e] << 16), b = __uint_as_float(wv[e] & 0xffff0000u);
                n2 = fmaf(a, a, fmaf(b, b, n2));
            }
            n2 += __shfl_xor_sync(0xffffffffu, n2, 1);
            n2 += __shfl_xor_sync(0xffffffffu, n2, 2);
            n2 += __shfl_xor_sync(0xffffffffu, n2, 4);
            const size_t r = r0 + 4 * u + (lane >> 3);
            if (sub == 0 && r < rows) kw[r] = expf(n2 * expf(-tau[(r / p.N) % p.H]));
        }
    }
}

// dW over the batch, in a fixed order (deterministic).  Nonstationary: the partials hold
// dU (rows < M) and dV (rows >= M); dW1 = (dU + dV)/2, dW2 = (dU - dV)/2.
__global__ void dw_reduce_kernel(Problem p, const float* part, float* dW1, float* dW2,
                                 const float* dtau_part, float* dtau)
{
    const int d = p.d, M = p.M, Mc = p.nonstat ? 2 * M : M;
    const size_t per = (size_t)M * d;
    if (dtau && blockIdx.x == 0)  // dtau[h] = sum over the batch, in order
        for (int h = threadIdx.x; h < p.H; h += blockDim.x) {
            float t = 0.f;
            for (int bb = 0; bb < p.B; ++bb) t += dtau_part[(size_t)bb * p.H + h];
            dtau[h] = t;
        }
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < (size_t)p.H * per;
         idx += (size_t)gridDim.x * blockDim.x) {
        int h = (int)(idx / per);
        size_t e = idx % per;
        float a = 0.f, b = 0.f;
        for (int bb = 0; bb < p.B; ++bb) {
            const float* pp = part + ((size_t)bb * p.H + h) * Mc * d;
            a += pp[e];
            if (p.nonstat) b += pp[per + e];
        }
        if (!p.nonstat) {
            dW1[idx] = a;
        } else {
            dW1[idx] = 0.5f * (a + b);
            dW2[idx] = 0.5f * (a - b);
        }
    }
}

}  // namespace

size_t simt_fwd_smem_bytes(const Problem& p, int chunk)
{
    return fwd_layout(p, chunk).total * sizeof(float);
}

size_t simt_bwd_smem_bytes(const Problem& p, int chunk)
{
    return bwd_layout(p, chunk).total * sizeof(float);
}

static const size_t kSmemLimit = 227 * 1024;

int simt_pick_chunk_fwd(const Problem& p)
{
    for (int c : {32, 16, 8})
        if (simt_fwd_smem_bytes(p, c) <= kSmemLimit) return c;
    return 0;
}

int simt_pick_chunk_bwd(const Problem& p)
{
    const int Mc = p.nonstat ? 2 * p.M : p.M;
    if ((size_t)Mc * p.d > (size_t)kThreads * kMaxDwPerThread) return 0;
    for (int c : {32, 16, 8})
        if (simt_bwd_smem_bytes(p, c) <= kSmemLimit) return c;
    return 0;
}

// dW partials [B*H][Mc][d], then dtau partials [B*H].
size_t simt_bwd_ws_bytes(const Problem& p)
{
    const int Mc = p.nonstat ? 2 * p.M : p.M;
    return (size_t)p.B * p.H * (Mc * p.d + 1) * sizeof(float);
}

cudaError_t launch_key_weights(const Problem& p, const void* k, const float* tau, float* kw,
                               cudaStream_t s)
{
    const size_t rows = (size_t)p.B * p.H * p.N;
    if (p.bf16 && p.d == 64) {  // 16 rows per warp and iteration, 8 warps per block
        const int blocks = (int)std::min<size_t>((rows + 127) / 128, 152 * 16);
        key_weights_bf16_d64_kernel<<<blocks, kThreads, 0, s>>>(p, (const __nv_bfloat16*)k, tau,
                                                                 kw);
        return cudaGetLastError();
    }
    const int blocks = (int)std::min<size_t>((rows + kThreads - 1) / kThreads, 152 * 16);
    if (p.bf16)
        key_weights_kernel<<<blocks, kThreads, 0, s>>>(p, (const __nv_bfloat16*)k, tau, kw);
    else
        key_weights_kernel<<<blocks, kThreads, 0, s>>>(p, (const float*)k, tau, kw);
    return cudaGetLastError();
}

cudaError_t launch_featmap(const Problem& p, const void* x, const float* W1, const float* W2,
                           void* phi, cudaStream_t s)
{
    return launch_featmap_scaled(p, x, W1, W2, nullptr, phi, s);
}

cudaError_t launch_featmap_scaled(const Problem& p, const void* x, const float* W1,
                                  const float* W2, const float* rowscale, void* phi,
                                  cudaStream_t s)
{
    const size_t work = (size_t)p.B * p.H * p.N * p.M;
    const int blocks = (int)std::min<size_t>((work + kThreads - 1) / kThreads, 152 * 16);
    const float scale = 1.0f / sqrtf((float)p.M);
    if (p.bf16)
        featmap_kernel<<<blocks, kThreads, 0, s>>>(p, (const __nv_bfloat16*)x, W1, W2,
                                                   (__nv_bfloat16*)phi, scale, rowscale);
    else
        featmap_kernel<<<blocks, kThreads, 0, s>>>(p, (const float*)x, W1, W2, (float*)phi,
                                                   scale, rowscale);
    return cudaGetLastError();
}

cudaError_t launch_simt_fwd(const Problem& p, const void* q, const void* k, const void* v,
                            const float* W1, const float* W2, const float* tau, void* out,
                            float* den, cudaStream_t s)
{
    const int C = simt_pick_chunk_fwd(p);
    const size_t smem = simt_fwd_smem_bytes(p, C);
    const int grid = p.B * p.H;
    if (p.bf16) {
        auto kern = simt_fwd_kernel<__nv_bfloat16>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, kThreads, smem, s>>>(p, C, (const __nv_bfloat16*)q,
                                          (const __nv_bfloat16*)k, (const __nv_bfloat16*)v, W1,
                                          W2, tau, (__nv_bfloat16*)out, den);
    } else {
        auto kern = simt_fwd_kernel<float>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, kThreads, smem, s>>>(p, C, (const float*)q, (const float*)k,
                                          (const float*)v, W1, W2, tau, (float*)out, den);
    }
    return cudaGetLastError();
}

cudaError_t launch_simt_bwd(const Problem& p, const void* q, const void* k, const void* v,
                            const float* W1, const float* W2, const float* tau,
                            const void* out, const float* den, const void* dout, void* dq,
                            void* dk, void* dv, float* dW1, float* dW2, float* dtau,
                            void* scratch, cudaStream_t s)
{
    const int C = simt_pick_chunk_bwd(p);
    const size_t smem = simt_bwd_smem_bytes(p, C);
    const int grid = p.B * p.H;
    const int Mc = p.nonstat ? 2 * p.M : p.M;
    float* part = (float*)scratch;
    float* tpart = part + (size_t)p.B * p.H * Mc * p.d;
    if (p.bf16) {
        typedef __nv_bfloat16 T;
        auto kern = simt_bwd_kernel<T>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, kThreads, smem, s>>>(p, C, (const T*)q, (const T*)k, (const T*)v, W1, W2,
                                          tau, (const T*)out, den, (const T*)dout, (T*)dq,
                                          (T*)dk, (T*)dv, part, tpart);
    } else {
        typedef float T;
        auto kern = simt_bwd_kernel<T>;
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        kern<<<grid, kThreads, smem, s>>>(p, C, (const T*)q, (const T*)k, (const T*)v, W1, W2,
                                          tau, (const T*)out, den, (const T*)dout, (T*)dq,
                                          (T*)dk, (T*)dv, part, tpart);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const size_t work = (size_t)p.H * p.M * p.d;
    const int blocks = (int)std::min<size_t>((work + kThreads - 1) / kThreads, 152 * 8);
    dw_reduce_kernel<<<blocks, kThreads, 0, s>>>(p, part, dW1, dW2, tpart, tau ? dtau : nullptr);
    return cudaGetLastError();
}

}  // namespace flex
