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
#include <cuda.h>
#include <cuda_bf16.h>

#include <algorithm>

#include "flex_internal.h"
#include "tc_common.cuh"
#include "tc_util.cuh"

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

// sin and cos of x: Cody-Waite reduction by 2 pi to |r| <= pi (tc::reduce_2pi), then the
// hardware approximations, whose absolute error on [-pi, pi] is a few 1e-7.
__device__ __forceinline__ void sincos_reduced(float x, float* s, float* c)
{
    __sincosf(tc::reduce_2pi(x), s, c);
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

// The same features on the tensor cores for bf16 token vectors with d = 64: one CTA per
// (head, 128 sequences, q or k, group of 64 frequencies); the 128 rows arrive by TMA (a
// strided view of [B][H][64]); the projection x W^T runs on tcgen05 with W split into
// bf16 high and low parts (x is exactly bf16, so the two MMAs give the fp32 product to
// about 2^-17) into 64 (s) or 128 (n) tensor-memory columns; every thread takes one
// sequence and 32 frequencies: sin/cos after the reduction by 2 pi, for k the key weight
// of the norm prefactor from its row in shared memory, fp32 phi to the workspace.
template <bool NS, int G>
__global__ void __launch_bounds__(256)
    decode_features_tc(const __grid_constant__ CUtensorMap tmap_q,
                       const __grid_constant__ CUtensorMap tmap_k, int B, int H, int M,
                       const float* __restrict__ W1, const float* __restrict__ W2,
                       const float* __restrict__ tau, float* __restrict__ phi, int* status)
{
    using namespace tc;
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
    constexpr int P = NS ? 128 : 64;
    constexpr uint32_t X = 0, WH = 16384, WL = WH + P * 128;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sb = smem_u32(sm);
    __shared__ uint32_t tmem_base_sh;
    __shared__ __align__(8) uint64_t mbar, tma_bar;
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wg = warp >> 2, quad = warp & 3, t = 32 * quad + lane;
    const int nblk = (B + 127) / 128;
    int u = blockIdx.x;
    const int g = u % G; u /= G;
    const int which = u % 2; u /= 2;  // 0: q, 1: k
    const int blk = u % nblk, h = u / nblk, b0 = blk * 128;

    stage_freq_rows_split<NS, 1, 256>(sb + WH, sb + WL, W1, W2, h, M, tid, 64 * g);
    if (tid == 0) {
        mbar_init(&mbar, 1);
        mbar_init(&tma_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
        mbar_arrive_expect_tx(&tma_bar, kTileBytes);
        tma_load_3d(sb + X, which ? &tmap_k : &tmap_q, 0, h, b0, &tma_bar);
    }
    if (warp == 0) {
        tmem_alloc(&tmem_base_sh, P);
        tmem_relinquish();
    }
    fence_proxy_async();
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tm = tmem_base_sh;
    const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);

    bool ok = bar_wait(&tma_bar, 0, &abort_flag, status);
    ok = !__syncthreads_or(!ok);
    if (ok) {
        fence_after_sync();
        if (tid == 0) {
            constexpr uint32_t I_PROJ = idesc_bf16(128, P, 0, 0);
            const uint64_t dX = sdesc(sb + X, 16, 1024);
            const uint64_t dH = sdesc(sb + WH, 16, 1024), dL = sdesc(sb + WL, 16, 1024);
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
                mma_bf16(tm, dX + ((ks * 32) >> 4), dH + ((ks * 32) >> 4), I_PROJ, ks > 0);
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
                mma_bf16(tm, dX + ((ks * 32) >> 4), dL + ((ks * 32) >> 4), I_PROJ, 1u);
            mma_commit(&mbar);
        }
        ok = bar_wait(&mbar, 0, &abort_flag, status);
        ok = !__syncthreads_or(!ok);
    }
    if (ok) {
        fence_after_sync();
        const int b = b0 + t, F = 2 * M;
        const bool valid = b < B;
        float wsc = rsqrtf((float)M);
        if (which == 1 && tau) {  // key weight exp(|k|^2 exp(-tau)) from this k row
            float n2 = 0.f;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const uint4 q4 = *reinterpret_cast<const uint4*>(sm + X + swz128(t, 8 * c));
                const uint32_t wv[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float lo = __uint_as_float(wv[e] << 16), hi = __uint_as_float(wv[e] & 0xffff0000u);
                    n2 = fmaf(lo, lo, fmaf(hi, hi, n2));
                }
            }
            wsc *= expf(n2 * expf(-tau[h]));
        }
        float a[32], w[32];
        const uint32_t col = tm_row + 32 * wg;
        tmem_ld16(col, *reinterpret_cast<float(*)[16]>(&a[0]));
        tmem_ld16(col + 16, *reinterpret_cast<float(*)[16]>(&a[16]));
        if (NS) {
            tmem_ld16(col + 64, *reinterpret_cast<float(*)[16]>(&w[0]));
            tmem_ld16(col + 80, *reinterpret_cast<float(*)[16]>(&w[16]));
        }
        tmem_wait_ld();
        float pc[32], ps[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            float su, cu, sw, cw = 1.f;
            sincos_reduced(a[i], &su, &cu);
            if (NS) sincos_reduced(w[i], &sw, &cw);
            pc[i] = cu * cw * wsc;
            ps[i] = su * cw * wsc;
        }
        if (valid) {
            float* dst = phi + (((size_t)b * H + h) * 2 + which) * F + 64 * g + 32 * wg;
            float4* dc = reinterpret_cast<float4*>(dst);
            float4* ds = reinterpret_cast<float4*>(dst + M);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                dc[j] = make_float4(pc[4 * j], pc[4 * j + 1], pc[4 * j + 2], pc[4 * j + 3]);
                ds[j] = make_float4(ps[4 * j], ps[4 * j + 1], ps[4 * j + 2], ps[4 * j + 3]);
            }
        }
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == 0) tmem_dealloc(tm, P);
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

template <bool NS, int G>
cudaError_t launch_features_tc(const Problem& p, const void* q, const void* k, const float* W1,
                               const float* W2, const float* tau, float* phi, int* status,
                               cudaStream_t s)
{
    CUtensorMap mq, mk;
    if (!tc::make_head_rows_map(&mq, q, p.B, p.H) || !tc::make_head_rows_map(&mk, k, p.B, p.H))
        return cudaErrorInvalidValue;
    constexpr int P = NS ? 128 : 64;
    const int smem = 16384 + 2 * P * 128 + 1024;
    auto kern = decode_features_tc<NS, G>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const long long ctas = (long long)p.H * ((p.B + 127) / 128) * 2 * G;
    if (ctas > 0x7fffffffLL) return cudaErrorInvalidValue;
    kern<<<(unsigned)ctas, 256, smem, s>>>(mq, mk, p.B, p.H, p.M, W1, W2, tau, phi, status);
    return cudaGetLastError();
}

template <typename T, bool NS>
cudaError_t launch_typed(const Problem& p, const void* q, const void* k, const void* v,
                         const float* W1, const float* W2, const float* tau, float* S,
                         float* z, void* out, float* den, float* phi, int* status,
                         cudaStream_t s)
{
    const long long fctas = (long long)p.H * ((p.B + kG - 1) / kG) * ((p.M + kTF - 1) / kTF);
    const long long sctas = (long long)p.B * p.H;
    if (fctas > 0x7fffffffLL || sctas > 0x7fffffffLL) return cudaErrorInvalidValue;

    cudaError_t e;
    if (p.bf16 && p.d == 64 && (p.M == 64 || p.M == 128)) {  // tensor-core features
        e = p.M == 64 ? launch_features_tc<NS, 1>(p, q, k, W1, W2, tau, phi, status, s)
                      : launch_features_tc<NS, 2>(p, q, k, W1, W2, tau, phi, status, s);
        if (e != cudaSuccess) return e;
    } else {
        const size_t fsmem =
            ((size_t)kTF * (p.d + 4) * 2 + 2 * kG * p.d + 2 * kG) * sizeof(float);
        auto fk = p.d == 32    ? decode_features<T, NS, 8>
                  : p.d == 64  ? decode_features<T, NS, 16>
                  : p.d == 128 ? decode_features<T, NS, 32>
                               : decode_features<T, NS, 0>;
        e = cudaFuncSetAttribute(fk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)fsmem);
        if (e != cudaSuccess) return e;
        fk<<<(unsigned)fctas, kThreadsF, fsmem, s>>>(p.B, p.H, p.d, p.M, (const T*)q,
                                                    (const T*)k, W1, W2, tau, phi);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }

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
                          float* z, void* out, float* den, void* scratch, int* status,
                          cudaStream_t s)
{
    float* phi = (float*)scratch;
    if (p.bf16)
        return p.nonstat ? launch_typed<__nv_bfloat16, true>(p, q, k, v, W1, W2, tau, S, z, out,
                                                             den, phi, status, s)
                         : launch_typed<__nv_bfloat16, false>(p, q, k, v, W1, W2, tau, S, z,
                                                              out, den, phi, status, s);
    return p.nonstat
               ? launch_typed<float, true>(p, q, k, v, W1, W2, tau, S, z, out, den, phi, status, s)
               : launch_typed<float, false>(p, q, k, v, W1, W2, tau, S, z, out, den, phi, status,
                                            s);
}

}  // namespace flex
