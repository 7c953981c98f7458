// Causal forward of RFF linear attention on the 5th-generation tensor cores (tcgen05).
//
// Chunked scan of Eq. (linear att) with j <= i: the sequence is cut into chunks of 128
// tokens; inside a chunk the masked kernel matrix A = phi(Q) phi(K)^T is applied directly
// (A V), across chunks the running state S = sum phi(k) v^T and z = sum phi(k) carries the
// prefix (phi(Q) S, phi(Q) z).  phi never leaves the SM: the projection x W^T lands in
// tensor memory, the CUDA cores turn it into cos/sin features (Eq. phi_n, or the product
// form of Eq. phi_non) and write them as bf16 MMA operands to shared memory.
//
// Features are processed in groups of 64 frequencies (128 features: 64 cos + 64 sin);
// A, phi(Q) S and phi(Q) z accumulate over the groups, S and z are held per group.
// Features are unscaled ([cos, sin] instead of M^{-1/2}[cos, sin]); the factor cancels in
// the output and only the stored denominator is rescaled (den = den' / M).
//
// One CTA (256 threads, 8 warps) per (b, h) sequence.  Thread 0 issues every MMA; all
// threads take part in the CUDA-core phases.  Warps w and w+4 share TMEM lane quadrant
// w % 4 and split the columns.
//
// Tensor memory (512 columns x 128 lanes, fp32):
//   [0,128)    projection of one group (s: 64 cols a; n: 64 cols u, 64 cols w)
//   [128,256)  A = phi(Q) phi(K)^T of the chunk (row = query, col = key)
//   [256,320)  numerator phi(Q) S + A V           [320,336) phi(Q) z (column 0)
//   [336,336+64G)  S per group (lane = feature)   then 16 columns of z per group
#include "flex_internal.h"
#include "tc_common.cuh"

namespace flex {
namespace {
using namespace tc;

constexpr int kC = 128;   // tokens per chunk = MMA M
constexpr int kThreadsTC = 256;
constexpr long long kWaitCycles = 4000000000LL;  // ~2 s at 2 GHz: a bounded wait

template <bool NS, int G>
struct Cfg {
    static constexpr int P = NS ? 128 : 64;  // projection columns per group
    // shared memory offsets (bytes, 1024-aligned)
    static constexpr uint32_t Q = 0, K = 16384, V = 32768;
    static constexpr uint32_t W = 49152;
    static constexpr uint32_t PQ = W + G * P * 128;
    static constexpr uint32_t PK = PQ + 32768;
    static constexpr uint32_t S = PK + 32768;
    static constexpr uint32_t Z = S + G * 16384;
    static constexpr uint32_t ONES = Z + G * 4096;
    static constexpr uint32_t A = ONES + 4096;
    static constexpr uint32_t RS = A + 32768;
    static constexpr uint32_t BYTES = RS + 1024;
    // tensor memory columns
    static constexpr uint32_t T_P = 0, T_A = 128, T_O = 256, T_DN = 320, T_S = 336;
    static constexpr uint32_t T_Z = T_S + 64 * G;
    static_assert(T_Z + 16 * G <= 512, "tensor memory budget");
    static_assert(BYTES + 1024 <= 232448, "shared memory budget");
};

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d)
{
    asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(a), "r"(b), "r"(c),
                 "r"(d)
                 : "memory");
}

// Waits for one MMA commit phase; the CTA agrees on the outcome (false = gave up).
__device__ __forceinline__ bool wait_mma(uint64_t* mbar, uint32_t& phase, int* status)
{
    bool ok = false;
    const long long t0 = clock64();
    while (true) {
        if (mbar_try_wait(mbar, phase)) { ok = true; break; }
        if (clock64() - t0 > kWaitCycles) break;
    }
    phase ^= 1u;
    if (!ok && (threadIdx.x & 31) == 0) atomicExch(status, (int)FLEX_ETIMEOUT);
    const bool all_ok = !__syncthreads_or(!ok);
    fence_after_sync();
    return all_ok;
}

// Every thread: make its shared-memory writes visible to the tensor core and its tensor
// memory reads complete, then meet the others.
__device__ __forceinline__ void handoff_to_mma()
{
    fence_proxy_async();
    fence_before_sync();
    __syncthreads();
}

// Load rows [0, rows) of a [128 x 64] bf16 tile (row stride 64 elements) into a 128B-
// swizzled shared tile; rows >= rows_valid are zero-filled.
__device__ __forceinline__ void load_tile(const __nv_bfloat16* src, int rows_valid,
                                          uint32_t dst)
{
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int idx = threadIdx.x + kThreadsTC * i;
        const int r = idx >> 3, c = idx & 7;
        uint4 val = make_uint4(0, 0, 0, 0);
        if (r < rows_valid) val = __ldg(reinterpret_cast<const uint4*>(src + r * 64 + c * 8));
        st_shared_v4(dst + swz128(r, c * 8), val.x, val.y, val.z, val.w);
    }
}

// Features of one group for one chunk: projection in TMEM -> bf16 phi tile (K-major,
// block 0 = cos features, block 1 = sin features).  Thread: row t, frequencies
// [32*wg, 32*wg + 32) of the group.
template <bool NS>
__device__ __forceinline__ void features_to_smem(uint32_t tm_row, int wg, int t, bool valid,
                                                 uint32_t dst)
{
    float a[32], w[32];
    tmem_ld16(tm_row + 32 * wg, *reinterpret_cast<float(*)[16]>(&a[0]));
    tmem_ld16(tm_row + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&a[16]));
    if (NS) {
        tmem_ld16(tm_row + 64 + 32 * wg, *reinterpret_cast<float(*)[16]>(&w[0]));
        tmem_ld16(tm_row + 64 + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&w[16]));
    }
    tmem_wait_ld();
    uint32_t pc[16], ps[16];
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        float s0, c0, s1, c1;
        __sincosf(a[2 * i], &s0, &c0);
        __sincosf(a[2 * i + 1], &s1, &c1);
        if (NS) {
            const float cw0 = __cosf(w[2 * i]), cw1 = __cosf(w[2 * i + 1]);
            c0 *= cw0; s0 *= cw0; c1 *= cw1; s1 *= cw1;
        }
        if (!valid) { c0 = s0 = c1 = s1 = 0.f; }
        pc[i] = pack_bf16(c0, c1);
        ps[i] = pack_bf16(s0, s1);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const uint32_t off = swz128(t, (4 * wg + j) * 8);
        st_shared_v4(dst + off, pc[4 * j], pc[4 * j + 1], pc[4 * j + 2], pc[4 * j + 3]);
        st_shared_v4(dst + 16384 + off, ps[4 * j], ps[4 * j + 1], ps[4 * j + 2], ps[4 * j + 3]);
    }
}

template <bool NS, int G>
__global__ void __launch_bounds__(kThreadsTC, 1)
    tc_fwd_causal_kernel(int H, int N, int M, const __nv_bfloat16* __restrict__ q,
                         const __nv_bfloat16* __restrict__ k,
                         const __nv_bfloat16* __restrict__ v, const float* __restrict__ W1,
                         const float* __restrict__ W2, __nv_bfloat16* __restrict__ out,
                         float* __restrict__ den, int* status)
{
    using L = Cfg<NS, G>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sb = smem_u32(sm);
    __shared__ uint32_t tmem_base_sh;
    __shared__ __align__(8) uint64_t mbar;
    float* rs = reinterpret_cast<float*>(sm + L::RS);  // [2][128] row sums of bf16(A)

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wg = warp >> 2, quad = warp & 3, t = 32 * quad + lane;
    const int bh = blockIdx.x, h = bh % H;
    const size_t base = (size_t)bh * N * 64;

    // ---- set-up: frequencies (bf16, K-major rows), zero state snapshots, ones ----
    for (int idx = tid; idx < G * L::P * 8; idx += kThreadsTC) {
        const int row = idx >> 3, c = idx & 7;
        const int g = row / L::P, r = row % L::P;
        const int f = 64 * g + (r & 63);
        const float* w1 = W1 + ((size_t)h * M + f) * 64 + c * 8;
        float x[8];
        if (!NS) {
#pragma unroll
            for (int e = 0; e < 8; ++e) x[e] = w1[e];
        } else {
            const float* w2 = W2 + ((size_t)h * M + f) * 64 + c * 8;
            const float sgn = r < 64 ? 1.f : -1.f;  // U = (W1+W2)/2, V = (W1-W2)/2
#pragma unroll
            for (int e = 0; e < 8; ++e) x[e] = 0.5f * (w1[e] + sgn * w2[e]);
        }
        st_shared_v4(sb + L::W + g * L::P * 128 + swz128(r, c * 8), pack_bf16(x[0], x[1]),
                     pack_bf16(x[2], x[3]), pack_bf16(x[4], x[5]), pack_bf16(x[6], x[7]));
    }
    for (int idx = tid; idx < (G * (16384 + 4096)) / 16; idx += kThreadsTC)
        st_shared_v4(sb + L::S + idx * 16, 0, 0, 0, 0);
    for (int idx = tid; idx < 4096 / 16; idx += kThreadsTC) {
        const uint32_t one2 = 0x3F803F80u;  // two bf16 ones
        st_shared_v4(sb + L::ONES + idx * 16, one2, one2, one2, one2);
    }
    if (tid == 0) {
        mbar_init(&mbar, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(&tmem_base_sh, 512);
        tmem_relinquish();
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tm = tmem_base_sh;
    const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);  // this warp's lane quadrant
    uint32_t phase = 0;

    constexpr uint32_t I_PROJ = idesc_bf16(128, L::P, 0, 0);
    constexpr uint32_t I_QK = idesc_bf16(128, 128, 0, 0);
    constexpr uint32_t I_QS = idesc_bf16(128, 64, 0, 1);
    constexpr uint32_t I_QZ = idesc_bf16(128, 16, 0, 0);
    constexpr uint32_t I_KV = idesc_bf16(128, 64, 1, 1);
    constexpr uint32_t I_K1 = idesc_bf16(128, 16, 1, 0);
    constexpr uint32_t I_AV = idesc_bf16(128, 64, 0, 1);

    const int nchunks = (N + kC - 1) / kC;
    for (int c = 0; c < nchunks; ++c) {
        const int t0 = c * kC, CL = min(kC, N - t0);
        const bool valid = t < CL;
        load_tile(q + base + (size_t)t0 * 64, CL, sb + L::Q);
        load_tile(k + base + (size_t)t0 * 64, CL, sb + L::K);
        load_tile(v + base + (size_t)t0 * 64, CL, sb + L::V);
        handoff_to_mma();

        for (int g = 0; g < G; ++g) {
            for (int which = 0; which < 2; ++which) {  // 0: q, 1: k
                if (tid == 0) {
                    fence_after_sync();
                    const uint32_t x0 = sb + (which ? L::K : L::Q);
                    const uint32_t w0 = sb + L::W + g * L::P * 128;
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        mma_bf16(tm + L::T_P, sdesc(x0 + ks * 32, 16, 1024),
                                 sdesc(w0 + ks * 32, 16, 1024), I_PROJ, ks > 0);
                    mma_commit(&mbar);
                }
                if (!wait_mma(&mbar, phase, status)) goto done;
                features_to_smem<NS>(tm_row + L::T_P, wg, t, valid,
                                     sb + (which ? L::PK : L::PQ));
                handoff_to_mma();
            }
            if (tid == 0) {
                fence_after_sync();
                const uint32_t pq = sb + L::PQ, pk = sb + L::PK;
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {  // K = 128 features of group g
                    const uint32_t kofs = (ks >> 2) * 16384 + (ks & 3) * 32;
                    const uint64_t aq = sdesc(pq + kofs, 16, 1024);
                    const uint32_t acc = (g > 0 || ks > 0) ? 1u : 0u;
                    mma_bf16(tm + L::T_A, aq, sdesc(pk + kofs, 16, 1024), I_QK, acc);
                    mma_bf16(tm + L::T_O, aq, sdesc(sb + L::S + g * 16384 + ks * 2048, 16384, 1024),
                             I_QS, acc);
                    mma_bf16(tm + L::T_DN, aq,
                             sdesc(sb + L::Z + g * 4096 + (ks >> 2) * 2048 + (ks & 3) * 32, 16,
                                   1024),
                             I_QZ, acc);
                }
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {  // K = 128 tokens of the chunk
                    const uint64_t ak = sdesc(pk + ks * 2048, 16384, 1024);
                    const uint32_t acc = (c > 0 || ks > 0) ? 1u : 0u;
                    mma_bf16(tm + L::T_S + 64 * g, ak, sdesc(sb + L::V + ks * 2048, 16384, 1024),
                             I_KV, acc);
                    mma_bf16(tm + L::T_Z + 16 * g, ak,
                             sdesc(sb + L::ONES + (ks >> 2) * 2048 + (ks & 3) * 32, 16, 1024),
                             I_K1, acc);
                }
                mma_commit(&mbar);
            }
            if (!wait_mma(&mbar, phase, status)) goto done;
        }

        // ---- A: causal mask, bf16, row sums; written as the K-major A operand of A V ----
        {
            float a[64];
#pragma unroll
            for (int j = 0; j < 4; ++j)
                tmem_ld16(tm_row + L::T_A + 64 * wg + 16 * j,
                          *reinterpret_cast<float(*)[16]>(&a[16 * j]));
            tmem_wait_ld();
            float sum = 0.f;
            uint32_t pk2[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                const int j0 = 64 * wg + 2 * i;
                const float x0 = (j0 <= t) ? a[2 * i] : 0.f;
                const float x1 = (j0 + 1 <= t) ? a[2 * i + 1] : 0.f;
                pk2[i] = pack_bf16(x0, x1);
                const __nv_bfloat162 b2 = *reinterpret_cast<__nv_bfloat162*>(&pk2[i]);
                sum += __bfloat162float(b2.x) + __bfloat162float(b2.y);
            }
#pragma unroll
            for (int cc = 0; cc < 8; ++cc)
                st_shared_v4(sb + L::A + wg * 16384 + swz128(t, cc * 8), pk2[4 * cc],
                             pk2[4 * cc + 1], pk2[4 * cc + 2], pk2[4 * cc + 3]);
            rs[wg * 128 + t] = sum;
        }
        handoff_to_mma();
        if (tid == 0) {
            fence_after_sync();
#pragma unroll
            for (int ks = 0; ks < 8; ++ks)
                mma_bf16(tm + L::T_O, sdesc(sb + L::A + (ks >> 2) * 16384 + (ks & 3) * 32, 16, 1024),
                         sdesc(sb + L::V + ks * 2048, 16384, 1024), I_AV, 1u);
            mma_commit(&mbar);
        }
        if (!wait_mma(&mbar, phase, status)) goto done;

        if (wg == 0) {
            // ---- output rows: out = num / den ----
            float o[64], dn[16];
#pragma unroll
            for (int j = 0; j < 4; ++j)
                tmem_ld16(tm_row + L::T_O + 16 * j, *reinterpret_cast<float(*)[16]>(&o[16 * j]));
            tmem_ld16(tm_row + L::T_DN, dn);
            tmem_wait_ld();
            const float dd = dn[0] + rs[t] + rs[128 + t];
            if (valid) {
                const float inv = 1.f / dd;
                uint4* dst = reinterpret_cast<uint4*>(out + base + (size_t)(t0 + t) * 64);
#pragma unroll
                for (int cc = 0; cc < 8; ++cc)
                    dst[cc] = make_uint4(pack_bf16(o[8 * cc] * inv, o[8 * cc + 1] * inv),
                                         pack_bf16(o[8 * cc + 2] * inv, o[8 * cc + 3] * inv),
                                         pack_bf16(o[8 * cc + 4] * inv, o[8 * cc + 5] * inv),
                                         pack_bf16(o[8 * cc + 6] * inv, o[8 * cc + 7] * inv));
                if (den) den[(size_t)bh * N + t0 + t] = dd / (float)M;
            }
        } else {
            // ---- state snapshot for the next chunk: S (MN-major rows) and z (K-major row 0) ----
#pragma unroll
            for (int g = 0; g < G; ++g) {
                float s[64], zz[16];
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    tmem_ld16(tm_row + L::T_S + 64 * g + 16 * j,
                              *reinterpret_cast<float(*)[16]>(&s[16 * j]));
                tmem_ld16(tm_row + L::T_Z + 16 * g, zz);
                tmem_wait_ld();
                const int f = t;  // feature within the group
#pragma unroll
                for (int cc = 0; cc < 8; ++cc)
                    st_shared_v4(sb + L::S + g * 16384 + swz128(f, cc * 8),
                                 pack_bf16(s[8 * cc], s[8 * cc + 1]),
                                 pack_bf16(s[8 * cc + 2], s[8 * cc + 3]),
                                 pack_bf16(s[8 * cc + 4], s[8 * cc + 5]),
                                 pack_bf16(s[8 * cc + 6], s[8 * cc + 7]));
                *reinterpret_cast<__nv_bfloat16*>(sm + L::Z + g * 4096 + (f >> 6) * 2048 +
                                                  swz128(0, f & 63)) = __float2bfloat16_rn(zz[0]);
            }
        }
        handoff_to_mma();
    }
done:
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == 0) tmem_dealloc(tm, 512);
}

template <bool NS, int G>
cudaError_t launch_one(const Problem& p, const void* q, const void* k, const void* v,
                       const float* W1, const float* W2, void* out, float* den, int* status,
                       cudaStream_t s)
{
    auto kern = tc_fwd_causal_kernel<NS, G>;
    const int smem = (int)Cfg<NS, G>::BYTES + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    kern<<<p.B * p.H, kThreadsTC, smem, s>>>(p.H, p.N, p.M, (const __nv_bfloat16*)q,
                                              (const __nv_bfloat16*)k, (const __nv_bfloat16*)v,
                                              W1, W2, (__nv_bfloat16*)out, den, status);
    return cudaGetLastError();
}

}  // namespace

bool tc_fwd_supported(const Problem& p)
{
    return p.bf16 && p.d == 64 && (p.M == 64 || p.M == 128) && p.causal;
}

cudaError_t launch_tc_fwd(const Problem& p, const void* q, const void* k, const void* v,
                          const float* W1, const float* W2, void* out, float* den, int* status,
                          cudaStream_t s)
{
    const int G = p.M / 64;
    if (p.nonstat)
        return G == 1 ? launch_one<true, 1>(p, q, k, v, W1, W2, out, den, status, s)
                      : launch_one<true, 2>(p, q, k, v, W1, W2, out, den, status, s);
    return G == 1 ? launch_one<false, 1>(p, q, k, v, W1, W2, out, den, status, s)
                  : launch_one<false, 2>(p, q, k, v, W1, W2, out, den, status, s);
}

}  // namespace flex
