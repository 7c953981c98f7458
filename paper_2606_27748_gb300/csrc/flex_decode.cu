// Recurrent decode step of causal RFF linear attention.
//
// Causal Eq. (linear att) as running sums: after token i, S_i = sum_{j<=i} phi(k_j) v_j^T
// and z_i = sum_{j<=i} phi(k_j), and out_i = phi(q_i)^T S_i / phi(q_i)^T z_i.  One call
// absorbs one new token per (b, h) into the caller's fp32 state and emits its output --
// the serving path of a causal model, one token at a time.
//
// The step is a stream over the state (2 x 2M x (d + 1) x 4 bytes per (b, h), read and
// written once); the feature map is a small batched product per head.  Two kernels:
//   decode_features  one CTA per (head, kG = 32 sequences, tile of 32 frequency rows):
//                    the tile is copied into shared memory and serves all 2 kG token
//                    vectors (q and k), so W is read 2 kG times less often than by a
//                    per-token kernel; phi(q), phi(k) (Eq. phi_n, or the product form of
//                    Eq. phi_non with u = (W1+W2)/2 x and w = (W1-W2)/2 x formed from the
//                    two dot products; scaled by M^{-1/2}; fp32, sin/cos after a
//                    reduction by 2 pi; phi(k) times the key weight exp(|k|^2 exp(-tau))
//                    of the norm prefactor when tau is given) go to the workspace;
//   decode_state     one CTA of 256 threads per (b, h), three per SM: starts asynchronous
//                    16-byte copies of S (up to 64 KB of rows) into shared memory and the
//                    loads of z, THEN waits for the features (programmatic dependent
//                    launch: the copies overlap the features kernel), updates
//                    S += phi(k) v^T, z += phi(k), stores them back, and forms
//                    out = phi(q)^T S / phi(q)^T z from the updated state with partials
//                    summed in a fixed order (bit-exact repeatable).  A state of more than
//                    64 KB per (b, h) (M d > 8192) goes through shared memory in row
//                    chunks.
#include <cuda_bf16.h>

#include <algorithm>

#include "flex_internal.h"

namespace flex {
namespace {

constexpr int kThreadsF = 256;
constexpr int kG = 32;         // sequences of one head per features CTA
constexpr int kTF = 32;        // frequency rows per shared-memory tile (one per lane)
constexpr int kThreadsD = 256;
constexpr int kSBuf = 16384;   // floats of S staged in shared memory per chunk (64 KB)
constexpr int kMaxF = 512;     // 2M, M <= 256
constexpr int kMaxD = 128;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem)
{
    const unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
// A load that stays after griddepcontrol.wait: volatile asm keeps its order relative to
// the wait (a plain load from a const __restrict__ pointer may be hoisted above it), and
// .cg reads L2, where the previous grid's stores are.
__device__ __forceinline__ float ld_after_wait(const float* p)
{
    float x;
    asm volatile("ld.global.cg.f32 %0, [%1];\n" : "=f"(x) : "l"(p) : "memory");
    return x;
}
__device__ __forceinline__ void cp_async_wait_all()
{
    asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;\n" ::: "memory");
}

// sin and cos of x: Cody-Waite reduction by 2 pi (the fp32 value of 2 pi plus the fp32
// value of the remainder, both computed from the mathematical constant) to |r| <= pi, then
// the hardware approximations, whose absolute error on [-pi, pi] is a few 1e-7.
__device__ __forceinline__ void sincos_reduced(float x, float* s, float* c)
{
    constexpr float kInv2Pi = 0.15915493667125702f;
    constexpr float k2PiHi = 6.2831854820251465f;
    constexpr float k2PiLo = -1.7484555314695172e-07f;
    const float n = rintf(x * kInv2Pi);
    const float r = fmaf(-n, k2PiLo, fmaf(-n, k2PiHi, x));
    __sincosf(r, s, c);
}

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }
__device__ __forceinline__ void from_f32(float* p, float x) { *p = x; }
__device__ __forceinline__ void from_f32(__nv_bfloat16* p, float x) { *p = __float2bfloat16_rn(x); }

// phi: [B*H][2][2M] fp32 (0 = phi(q), 1 = phi(k)).  CTA = (head, kG sequences, tile of
// kTF frequency rows); lane = row, warp = kTokW token vectors, so each thread carries
// 2 kTokW independent dot products (W1 x and W2 x of its rows).
// D4C: d / 4 as a compile-time constant (the inner loop unrolls fully), or 0 for any d.
template <typename T, bool NS, int D4C>
__global__ void __launch_bounds__(kThreadsF, 4)
    decode_features(int B, int H, int d, int M, const T* __restrict__ q,
                    const T* __restrict__ k, const float* __restrict__ W1,
                    const float* __restrict__ W2, const float* __restrict__ tau,
                    float* __restrict__ phi)
{
    // The state kernel may launch now; it waits for this grid before reading phi.
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    extern __shared__ float4 fsm4[];
    // Row pitch d + 4 floats: the float4 reads of 32 rows (one per lane) take the minimum
    // of 4 shared-memory wavefronts, and every row starts on 16 bytes.
    const int ld = D4C ? 4 * D4C + 4 : d + 4, F = 2 * M;
    float* w1s = reinterpret_cast<float*>(fsm4);  // [kTF][ld]: W1 rows of the tile
    float* w2s = w1s + kTF * ld;                  // [kTF][ld]: W2 rows (n only)
    float* xs = w2s + (NS ? kTF * ld : 0);        // [2 kG][d]: token vector t = 2 s + which
    float* kw = xs + 2 * kG * (D4C ? 4 * D4C : d); // [2 kG]: key weights (norm prefactor)
    const int tiles = (M + kTF - 1) / kTF, groups = (B + kG - 1) / kG;
    const int tile = blockIdx.x % tiles, grp = (blockIdx.x / tiles) % groups;
    const int h = blockIdx.x / (tiles * groups);
    const int b0 = grp * kG, f0 = tile * kTF, ntok = 2 * min(kG, B - b0);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int d4 = D4C ? D4C : d / 4, dd = 4 * d4;
    constexpr int kWarps = kThreadsF / 32;
    constexpr int kTokW = 2 * kG / kWarps;        // token vectors per warp
    constexpr int kXE = D4C ? (4 * D4C + 31) / 32 : kMaxD / 32;  // elements per lane and vector

    // Staging: the W tile by asynchronous copies (no registers), rows past M zero; the
    // token vectors through registers (bf16 -> fp32), all loads before the first store.
    for (int i = tid; i < kTF * d4; i += kThreadsF) {
        const int r = i / d4, e4 = i % d4, f = f0 + r;
        float4* d1 = reinterpret_cast<float4*>(w1s + r * ld) + e4;
        float4* d2 = reinterpret_cast<float4*>(w2s + r * ld) + e4;
        if (f < M) {
            cp_async16(d1, W1 + ((size_t)h * M + f) * dd + 4 * e4);
            if (NS) cp_async16(d2, W2 + ((size_t)h * M + f) * dd + 4 * e4);
        } else {
            *d1 = make_float4(0.f, 0.f, 0.f, 0.f);
            if (NS) *d2 = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    float xr[kTokW][kXE];
#pragma unroll
    for (int j = 0; j < kTokW; ++j) {             // warp per token vector, lane per element
        const int t = warp + j * kWarps;
        const size_t io = ((size_t)(b0 + t / 2) * H + h) * dd;
#pragma unroll
        for (int i = 0; i < kXE; ++i) {
            const int e = lane + 32 * i;
            xr[j][i] = (t < ntok && e < dd) ? to_f32((t & 1) ? k[io + e] : q[io + e]) : 0.f;
        }
    }
#pragma unroll
    for (int j = 0; j < kTokW; ++j)
#pragma unroll
        for (int i = 0; i < kXE; ++i)
            if (lane + 32 * i < dd) xs[(warp + j * kWarps) * dd + lane + 32 * i] = xr[j][i];
    cp_async_wait_all();
    __syncthreads();
    if (tau) {  // key weight of the norm prefactor (Sec. 3.2): exp(|k|^2 exp(-tau))
        if (tid < 2 * kG) {
            float n2 = 0.f;
            for (int e = 0; e < dd; ++e) n2 = fmaf(xs[tid * dd + e], xs[tid * dd + e], n2);
            kw[tid] = expf(n2 * expf(-tau[h]));
        }
        __syncthreads();
    }

    float a[kTokW], c[kTokW];
#pragma unroll
    for (int j = 0; j < kTokW; ++j) a[j] = c[j] = 0.f;
    const float4* r1 = reinterpret_cast<const float4*>(w1s + lane * ld);
    const float4* r2 = reinterpret_cast<const float4*>(w2s + lane * ld);
    const float4* x4 = reinterpret_cast<const float4*>(xs);
#pragma unroll(D4C ? D4C : 2)
    for (int e4 = 0; e4 < d4; ++e4) {
        const float4 p1 = r1[e4];
        const float4 p2 = NS ? r2[e4] : p1;
#pragma unroll
        for (int j = 0; j < kTokW; ++j) {
            const float4 xv = x4[(warp + j * kWarps) * d4 + e4];  // broadcast
            a[j] = fmaf(p1.x, xv.x, fmaf(p1.y, xv.y, fmaf(p1.z, xv.z, fmaf(p1.w, xv.w, a[j]))));
            if (NS)
                c[j] = fmaf(p2.x, xv.x, fmaf(p2.y, xv.y, fmaf(p2.z, xv.z, fmaf(p2.w, xv.w, c[j]))));
        }
    }
    const float scale = rsqrtf((float)M);
    const int f = f0 + lane;
#pragma unroll
    for (int j = 0; j < kTokW; ++j) {
        const int t = warp + j * kWarps;
        if (t < ntok && f < M) {
            // n: u = (W1 + W2)/2 x, w = (W1 - W2)/2 x; s: u = W1 x
            float su, cu, sw, cw = 1.f;
            sincos_reduced(NS ? 0.5f * (a[j] + c[j]) : a[j], &su, &cu);
            if (NS) sincos_reduced(0.5f * (a[j] - c[j]), &sw, &cw);
            cw *= scale;
            if (tau && (t & 1)) cw *= kw[t];  // phi(k) carries its weight into S and z
            float* dst = phi + (((size_t)(b0 + t / 2) * H + h) * 2 + (t & 1)) * F;
            dst[f] = cu * cw;
            dst[M + f] = su * cw;
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(kThreadsD, 3)
    decode_state(int d, int M, const T* __restrict__ v, const float* phi,
                 float* __restrict__ S, float* __restrict__ z, T* __restrict__ out,
                 float* __restrict__ den)
{
    extern __shared__ float4 sS[];                  // [rows of the chunk][d / 4]
    __shared__ __align__(16) float vs[kMaxD];
    __shared__ __align__(16) float ph[2][kMaxF];    // phi(q), phi(k)
    __shared__ float red[kThreadsD * 4];            // [row group][d] numerator partials
    __shared__ float dred[kThreadsD / 32];

    const int F = 2 * M, d4 = d / 4, tid = threadIdx.x;
    const size_t u = blockIdx.x;
    const int crows = min(F, kSBuf / d);            // rows per chunk
    float4* S4 = reinterpret_cast<float4*>(S + u * F * d);

    // state copies and loads first: they depend on nothing this step computes
    for (int i = tid; i < crows * d4; i += kThreadsD) cp_async16(sS + i, S4 + i);
    float* zu = z + u * F;
    float zr[kMaxF / kThreadsD];
#pragma unroll
    for (int j = 0; j < kMaxF / kThreadsD; ++j)
        if (tid + kThreadsD * j < F) zr[j] = zu[tid + kThreadsD * j];
    if (tid < d) vs[tid] = to_f32(v[u * d + tid]);

    asm volatile("griddepcontrol.wait;\n" ::: "memory");  // the features are written
    float pr[2 * kMaxF / kThreadsD];                        // all loads, then the stores
#pragma unroll
    for (int j = 0; j < 2 * kMaxF / kThreadsD; ++j)
        if (tid + kThreadsD * j < 2 * F) pr[j] = ld_after_wait(phi + u * 2 * F + tid + kThreadsD * j);
#pragma unroll
    for (int j = 0; j < 2 * kMaxF / kThreadsD; ++j) {
        const int i = tid + kThreadsD * j;
        if (i < 2 * F) ph[i / F][i % F] = pr[j];
    }

    // Thread (rg, c4) owns float4 column c4 of the rows rg + ngrp * i of each chunk.
    const int ngrp = kThreadsD / d4, rg = tid / d4, c4 = tid % d4;
    float4 num = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int r0 = 0; r0 < F; r0 += crows) {
        const int nr = min(crows, F - r0);
        if (r0 > 0) {
            __syncthreads();  // every thread is done with the previous chunk
            for (int i = tid; i < nr * d4; i += kThreadsD)
                cp_async16(sS + i, S4 + (size_t)r0 * d4 + i);
        }
        cp_async_wait_all();
        __syncthreads();
        if (rg < ngrp) {
            const float4 vv = reinterpret_cast<const float4*>(vs)[c4];
#pragma unroll 4
            for (int r = rg; r < nr; r += ngrp) {
                const float pk = ph[1][r0 + r], pq = ph[0][r0 + r];
                float4 s = sS[r * d4 + c4];
                s.x = fmaf(pk, vv.x, s.x);
                s.y = fmaf(pk, vv.y, s.y);
                s.z = fmaf(pk, vv.z, s.z);
                s.w = fmaf(pk, vv.w, s.w);
                S4[(size_t)(r0 + r) * d4 + c4] = s;
                num.x = fmaf(pq, s.x, num.x);
                num.y = fmaf(pq, s.y, num.y);
                num.z = fmaf(pq, s.z, num.z);
                num.w = fmaf(pq, s.w, num.w);
            }
        }
    }
    if (rg < ngrp) reinterpret_cast<float4*>(red)[rg * d4 + c4] = num;

    float dn = 0.f;
#pragma unroll
    for (int j = 0; j < kMaxF / kThreadsD; ++j) {
        const int f = tid + kThreadsD * j;
        if (f < F) {
            const float zz = zr[j] + ph[1][f];
            zu[f] = zz;
            dn = fmaf(ph[0][f], zz, dn);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dn += __shfl_xor_sync(0xffffffffu, dn, o);
    if ((tid & 31) == 0) dred[tid >> 5] = dn;
    __syncthreads();

    if (tid < d) {
        float nsum = 0.f, dsum = 0.f;
        for (int g = 0; g < ngrp; ++g) nsum += red[g * d + tid];  // fixed order
#pragma unroll
        for (int w = 0; w < kThreadsD / 32; ++w) dsum += dred[w];
        from_f32(out + u * d + tid, nsum / dsum);
        if (den && tid == 0) den[u] = dsum;
    }
}

template <typename T, bool NS>
cudaError_t launch_typed(const Problem& p, const void* q, const void* k, const void* v,
                         const float* W1, const float* W2, const float* tau, float* S,
                         float* z, void* out, float* den, float* phi, cudaStream_t s)
{
    const long long fctas = (long long)p.H * ((p.B + kG - 1) / kG) * ((p.M + kTF - 1) / kTF);
    const long long sctas = (long long)p.B * p.H;
    if (fctas > 0x7fffffffLL || sctas > 0x7fffffffLL) return cudaErrorInvalidValue;

    const size_t fsmem = ((size_t)kTF * (p.d + 4) * 2 + 2 * kG * p.d + 2 * kG) * sizeof(float);
    auto fk = p.d == 32    ? decode_features<T, NS, 8>
              : p.d == 64  ? decode_features<T, NS, 16>
              : p.d == 128 ? decode_features<T, NS, 32>
                           : decode_features<T, NS, 0>;
    cudaError_t e = cudaFuncSetAttribute(fk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)fsmem);
    if (e != cudaSuccess) return e;
    fk<<<(unsigned)fctas, kThreadsF, fsmem, s>>>(p.B, p.H, p.d, p.M, (const T*)q, (const T*)k,
                                                W1, W2, tau, phi);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;

    const size_t ssmem = (size_t)std::min(2 * p.M, kSBuf / p.d) * p.d * sizeof(float);
    auto sk = decode_state<T>;
    if ((e = cudaFuncSetAttribute(sk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ssmem)) !=
        cudaSuccess)
        return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)sctas);
    cfg.blockDim = dim3(kThreadsD);
    cfg.dynamicSmemBytes = ssmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, sk, p.d, p.M, (const T*)v, (const float*)phi, S, z, (T*)out,
                              den);
}

}  // namespace

size_t decode_ws_bytes(const Problem& p) { return (size_t)p.B * p.H * 2 * 2 * p.M * sizeof(float); }

cudaError_t launch_decode(const Problem& p, const void* q, const void* k, const void* v,
                          const float* W1, const float* W2, const float* tau, float* S,
                          float* z, void* out, float* den, void* scratch, cudaStream_t s)
{
    float* phi = (float*)scratch;
    if (p.bf16)
        return p.nonstat ? launch_typed<__nv_bfloat16, true>(p, q, k, v, W1, W2, tau, S, z, out,
                                                             den, phi, s)
                         : launch_typed<__nv_bfloat16, false>(p, q, k, v, W1, W2, tau, S, z,
                                                              out, den, phi, s);
    return p.nonstat ? launch_typed<float, true>(p, q, k, v, W1, W2, tau, S, z, out, den, phi, s)
                     : launch_typed<float, false>(p, q, k, v, W1, W2, tau, S, z, out, den, phi, s);
}

}  // namespace flex
