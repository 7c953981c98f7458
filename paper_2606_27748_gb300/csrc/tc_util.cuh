// Helpers shared by the tensor-core kernels: bf16 packing, vector shared stores, bounded
// mbarrier waits with a CTA-wide abort flag, and host-side TMA descriptor creation.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>

#include "flex_internal.h"
#include "tc_common.cuh"

namespace flex {
namespace tc {

constexpr long long kWaitCycles = 4000000000LL;  // ~2 s at 2 GHz: every wait is bounded
constexpr uint32_t kTileBytes = 128 * 128;       // one 128 x 64 bf16 tile

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

// ---- sin/cos arguments ----------------------------------------------------------------
// The hardware sin/cos (MUFU, reached through __sincosf / __cosf) is accurate to about
// 2^-21 absolute on [-pi, pi]; beyond it the error grows with |x| (measured on GB300 over
// 2^16 points per range: 2^-19.6 for |x| <= 10, 2^-17.8 for |x| <= 30, 2^-12.9 for
// |x| <= 1000).  Projection values reach that range once the frequencies are trained
// (Sec. 3.2: the spectral frequencies are learned), so arguments are first reduced by
// 2 pi with a two-constant Cody-Waite step: n = rint(x / 2 pi), r = (x - n C1) - n C2,
// C1 the fp32 value of 2 pi and C2 the fp32 value of 2 pi - C1, each fma rounding once;
// measured after the reduction: 2^-21 for every |x| <= 2000.
constexpr float kPi = 3.14159265358979f;
constexpr float kInv2Pi = 0.15915493667125702f;
constexpr float k2PiHi = 6.2831854820251465f;
constexpr float k2PiLo = -1.7484555314695172e-07f;

__device__ __forceinline__ float reduce_2pi(float x)
{
    const float n = rintf(x * kInv2Pi);
    return fmaf(-n, k2PiLo, fmaf(-n, k2PiHi, x));
}

template <int n>
__device__ __forceinline__ void reduce_2pi_all(float (&v)[n])
{
#pragma unroll
    for (int i = 0; i < n; ++i) v[i] = reduce_2pi(v[i]);
}

// The range test: `mabs` is this thread's max |x| over its arguments, as the tensor-memory
// load returns it (tmem_ld16_maxabs).  Reduces every value of a (and of w) when any lane of
// the warp holds one with |x| >= 2 (or not finite); inside [-2, 2] (a subset of [-pi, pi],
// where the hardware sin/cos keeps its 2^-21 bound) the step is skipped for one compare and
// one vote.  Warp-collective: all 32 lanes call it together.
template <int n>
__device__ __forceinline__ void reduce_2pi_if_needed(float (&a)[n], float mabs)
{
    if (__any_sync(0xffffffffu, !(mabs < 2.f))) reduce_2pi_all(a);
}
template <int n>
__device__ __forceinline__ void reduce_2pi_if_needed(float (&a)[n], float (&w)[n], float mabs)
{
    if (__any_sync(0xffffffffu, !(mabs < 2.f))) {
        reduce_2pi_all(a);
        reduce_2pi_all(w);
    }
}

// ---- packed f32x2 arithmetic (two fp32 lanes in one 64-bit register) --------------------
__device__ __forceinline__ uint64_t f2_pack(float lo, float hi)
{
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void f2_unpack(uint64_t v, float& lo, float& hi)
{
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t f2_mul(uint64_t a, uint64_t b)
{
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c)
{
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}

// cos(x) for |x| <= 2 on the FMA pipe: p(x^2) with p of degree 4, fitted here to
// cos(sqrt(y)) on y in [0, 4] by least squares on 4000 Chebyshev nodes refined by Lawson's
// iteratively reweighted least squares (an approximation to the minimax polynomial);
// max error with fp32 evaluation 6.6e-7 over [-2, 2] (the hardware cos: 4e-7 on
// [-pi, pi]).  Two values per call, one packed multiply and four packed fmas.
__device__ __forceinline__ void cos_poly2(float& x0, float& x1)
{
    constexpr float C0 = 0.9999995231628418f, C1 = -0.4999936819076538f,
                    C2 = 0.04165392369031906f, C3 = -0.0013798808213323355f,
                    C4 = 2.2181484382599592e-05f;
    const uint64_t x = f2_pack(x0, x1), y = f2_mul(x, x);
    uint64_t p = f2_fma(f2_pack(C4, C4), y, f2_pack(C3, C3));
    p = f2_fma(p, y, f2_pack(C2, C2));
    p = f2_fma(p, y, f2_pack(C1, C1));
    p = f2_fma(p, y, f2_pack(C0, C0));
    f2_unpack(p, x0, x1);
}

// Nonstationary feature arguments u (a) and w, with mabs the max |x| over both: when any
// lane holds one with |x| >= 2 (or not finite), both are reduced and w is replaced by the
// hardware cos(w); otherwise w is replaced by cos(w) from the FMA-pipe polynomial.  Either
// way w holds cos(w) afterwards and a is ready for the hardware sin/cos.  Warp-collective.
template <int n>
__device__ __forceinline__ void cos_w_args(float (&a)[n], float (&w)[n], float mabs)
{
    static_assert(n % 2 == 0, "pairs");
    if (__any_sync(0xffffffffu, !(mabs < 2.f))) {
        reduce_2pi_all(a);
#pragma unroll
        for (int i = 0; i < n; ++i) w[i] = __cosf(reduce_2pi(w[i]));
    } else {
#pragma unroll
        for (int i = 0; i < n / 2; ++i) cos_poly2(w[2 * i], w[2 * i + 1]);
    }
}

// Bounded wait on one mbarrier phase.  On a time-out the CTA is told to stop (abort flag)
// and the status word (if any) records FLEX_ETIMEOUT; every other wait then returns at once.
__device__ __forceinline__ bool bar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                         int* status, long long limit = kWaitCycles)
{
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (clock64() - t0 > limit) {
            *abort_flag = 1;
            if (status) atomicExch(status, (int)FLEX_ETIMEOUT);
            return false;
        }
    }
}

// The diagnostic stall of flex_debug_stall: when the workspace header asks for it
// (stall_cycles > 0), one thread of the CTA waits that many clocks at most on `bar`, an
// mbarrier that nothing arrives on, so the wait runs out exactly as a wait for a lost
// arrival would: the abort flag is set and the status word records FLEX_ETIMEOUT.  Called
// during set-up, before anything is issued; the kernel then issues nothing and exits.
__device__ __forceinline__ void diagnostic_stall(uint64_t* bar, volatile int* abort_flag,
                                                 int* status)
{
    if (!status) return;
    const int cycles = *reinterpret_cast<volatile int*>(status + kStallWord);
    if (cycles > 0) bar_wait(bar, 0, abort_flag, status, cycles);
}

// On the way out after an abort: waits at most `limit` clocks, regardless of the abort
// flag, for a phase of an mbarrier that copies into this CTA's shared memory complete on,
// so that none is still in flight when the CTA exits.
constexpr long long kDrainCycles = 20000000LL;  // ~10 ms
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity, long long limit)
{
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity) && clock64() - t0 < limit) {
    }
}

// bar_wait for a barrier that other CTAs of the cluster arrive on (acquire at cluster scope).
__device__ __forceinline__ bool bar_wait_cluster(uint64_t* bar, uint32_t parity,
                                                 volatile int* abort_flag, int* status)
{
    const long long t0 = clock64();
    while (true) {
        if (mbar_try_wait_cluster(bar, parity)) return true;
        if (*abort_flag) return false;
        if (clock64() - t0 > kWaitCycles) {
            *abort_flag = 1;
            if (status) atomicExch(status, (int)FLEX_ETIMEOUT);
            return false;
        }
    }
}


// ---- host side ----------------------------------------------------------------------------

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

inline EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return (EncodeTiledFn) nullptr;
        return (EncodeTiledFn)p;
    }();
    return fn;
}

// [B*H][N][64] bf16 as a 3-D tensor; 128 x 64 boxes, 128-byte swizzle; rows past N read 0.
inline bool make_act_map(CUtensorMap* m, const void* base, int BH, int N)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {64, (cuuint64_t)N, (cuuint64_t)BH};
    cuuint64_t strides[2] = {128, (cuuint64_t)N * 128};
    cuuint32_t box[3] = {64, 128, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
               box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

// Output tiles of 32 rows x 32 columns of a [BH][N][64] bf16 tensor, 64-byte swizzle: in
// shared memory row r of a tile is 64 bytes at r * 64, its 16-byte chunk c stored at
// position c ^ ((r >> 1) & 3) (tile base 512-byte aligned).
inline bool make_out_map32(CUtensorMap* m, const void* base, int BH, int N)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {64, (cuuint64_t)N, (cuuint64_t)BH};
    cuuint64_t strides[2] = {128, (cuuint64_t)N * 128};
    cuuint32_t box[3] = {32, 32, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
               box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}
__host__ __device__ __forceinline__ uint32_t swz64(uint32_t row, uint32_t chunk)
{
    return row * 64 + ((chunk ^ ((row >> 1) & 3)) << 4);
}

// One head's frequency rows into shared memory, bf16, K-major with 128-byte swizzle: G
// groups of P rows (s: P = 64 rows of W1; n: P = 128, U = (W1+W2)/2 then V = (W1-W2)/2),
// row r of group g = frequency 64 g + r % 64.  8-float pieces by float4 loads, a batch of
// up to 4 pieces per thread in flight.  W1, W2: [H][M][64] fp32, 16-byte aligned.
template <bool NS, int G, int NTHREADS>
__device__ __forceinline__ void stage_freq_rows(uint32_t dst, const float* W1, const float* W2,
                                                int h, int M, int tid)
{
    constexpr int P = NS ? 128 : 64;
    static_assert(G * P * 8 % NTHREADS == 0, "whole pieces per thread");
    constexpr int kPieces = G * P * 8 / NTHREADS, kBatch = kPieces < 4 ? kPieces : 4;
    for (int i0 = 0; i0 < kPieces; i0 += kBatch) {
        float4 a[kBatch][2], c2[kBatch][2];
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            const int idx = tid + NTHREADS * (i0 + i), r = idx >> 3, c = idx & 7;
            const int f = 64 * (r / P) + ((r % P) & 63);
            const float4* w1 = reinterpret_cast<const float4*>(W1 + ((size_t)h * M + f) * 64 + c * 8);
            a[i][0] = __ldg(w1);
            a[i][1] = __ldg(w1 + 1);
            if (NS) {
                const float4* w2 = reinterpret_cast<const float4*>(W2 + ((size_t)h * M + f) * 64 + c * 8);
                c2[i][0] = __ldg(w2);
                c2[i][1] = __ldg(w2 + 1);
            }
        }
#pragma unroll
        for (int i = 0; i < kBatch; ++i) {
            const int idx = tid + NTHREADS * (i0 + i), r = idx >> 3, c = idx & 7;
            const float x0[8] = {a[i][0].x, a[i][0].y, a[i][0].z, a[i][0].w,
                                 a[i][1].x, a[i][1].y, a[i][1].z, a[i][1].w};
            float x[8];
            if (!NS) {
#pragma unroll
                for (int e = 0; e < 8; ++e) x[e] = x0[e];
            } else {
                const float y0[8] = {c2[i][0].x, c2[i][0].y, c2[i][0].z, c2[i][0].w,
                                     c2[i][1].x, c2[i][1].y, c2[i][1].z, c2[i][1].w};
                const float sgn = (r % P) < 64 ? 1.f : -1.f;
#pragma unroll
                for (int e = 0; e < 8; ++e) x[e] = 0.5f * (x0[e] + sgn * y0[e]);
            }
            st_shared_v4(dst + swz128(r, c * 8), pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]),
                         pack_bf16(x[4], x[5]), pack_bf16(x[6], x[7]));
        }
    }
}

// The same rows split into bf16 high and low parts (x = hi + lo to about 2^-17): hi at
// dst_hi, lo at dst_lo, both in the layout above; frequencies from f0 on.  Two MMAs (hi, lo) against an exactly
// representable bf16 operand reproduce the fp32 product to that accuracy.
template <bool NS, int G, int NTHREADS>
__device__ __forceinline__ void stage_freq_rows_split(uint32_t dst_hi, uint32_t dst_lo,
                                                      const float* W1, const float* W2, int h,
                                                      int M, int tid, int f0 = 0)
{
    constexpr int P = NS ? 128 : 64;
    static_assert(G * P * 8 % NTHREADS == 0, "whole pieces per thread");
    constexpr int kPieces = G * P * 8 / NTHREADS;
    for (int i = 0; i < kPieces; ++i) {
        const int idx = tid + NTHREADS * i, r = idx >> 3, c = idx & 7;
        const int f = f0 + 64 * (r / P) + ((r % P) & 63);
        const float4* w1 = reinterpret_cast<const float4*>(W1 + ((size_t)h * M + f) * 64 + c * 8);
        const float4 a0 = __ldg(w1), a1 = __ldg(w1 + 1);
        float x[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
        if (NS) {
            const float4* w2 = reinterpret_cast<const float4*>(W2 + ((size_t)h * M + f) * 64 + c * 8);
            const float4 b0 = __ldg(w2), b1 = __ldg(w2 + 1);
            const float y[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
            const float sgn = (r % P) < 64 ? 1.f : -1.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) x[e] = 0.5f * (x[e] + sgn * y[e]);
        }
        uint32_t hi[4], lo[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            hi[e] = pack_bf16(x[2 * e], x[2 * e + 1]);
            const float h0 = __uint_as_float(hi[e] << 16), h1 = __uint_as_float(hi[e] & 0xffff0000u);
            lo[e] = pack_bf16(x[2 * e] - h0, x[2 * e + 1] - h1);
        }
        st_shared_v4(dst_hi + swz128(r, c * 8), hi[0], hi[1], hi[2], hi[3]);
        st_shared_v4(dst_lo + swz128(r, c * 8), lo[0], lo[1], lo[2], lo[3]);
    }
}

// [BH][N][F] bf16 rows of F features (F a multiple of 64), box 64 x 128, 128B swizzle:
// a load at x = 64 g brings feature block g of 128 rows.
inline bool make_feat_map(CUtensorMap* m, const void* base, int BH, int N, int F)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)F, (cuuint64_t)N, (cuuint64_t)BH};
    cuuint64_t strides[2] = {(cuuint64_t)F * 2, (cuuint64_t)N * F * 2};
    cuuint32_t box[3] = {64, 128, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
               box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

// [B][H][64] bf16 token vectors of one step, viewed per head: box (64, 1 head, 128 batch
// entries), 128B swizzle: a load at (0, h, b0) brings 128 rows of head h.
inline bool make_head_rows_map(CUtensorMap* m, const void* base, int B, int H)
{
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {64, (cuuint64_t)H, (cuuint64_t)B};
    cuuint64_t strides[2] = {128, (cuuint64_t)H * 128};
    cuuint32_t box[3] = {64, 1, 128};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
               box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

inline int sm_count()
{
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    return n;
}

}  // namespace tc
}  // namespace flex
