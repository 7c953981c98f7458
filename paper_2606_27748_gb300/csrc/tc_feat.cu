// Feature map written out, on the tensor cores: phi(x) of Eq. phi_n (s) or the product
// form of Eq. phi_non (n) for every row of x [B*H*N][64] bf16, scaled by M^{-1/2} and by
// an optional per-row factor (the key weight of the norm prefactor), into
// phi [B*H*N][2M] bf16 (cos block, then sin block).
//
// One CTA per 4 blocks of 128 rows of one sequence (one head's frequencies, staged once),
// 256 threads: TMA loads the rows (the next block while the current one is worked on),
// thread 0 issues the projections x W^T (s: W1; n: U = (W1+W2)/2 and
// V = (W1-W2)/2), one group of 64 frequencies per 64 (s) or 128 (n) columns; every thread
// takes one row and 32 frequencies of each group: arguments reduced by 2 pi, hardware
// sin/cos, products, bf16 pack, 64-byte stores of its cos and sin runs.
//
// The frequencies enter the projection split into bf16 high and low parts (two MMAs into
// one fp32 accumulator): x is exactly bf16, so the projection carries the fp32
// frequencies to about 2^-17 instead of bf16's 2^-9.  The phase error of a single bf16
// rounding grows with the argument (|x . w| 2^-9), which would dominate the feature error
// once trained frequencies push arguments past ~10.
#include "flex_internal.h"
#include "tc_common.cuh"
#include "tc_util.cuh"

namespace flex {
namespace {
using namespace tc;

constexpr int kC = 128;
constexpr int kThreadsF = 256;
constexpr int kBlocksPerCta = 4;  // row blocks of one sequence per CTA (W staged once)

template <bool NS, int G>  // G = M / 64 frequency groups
__global__ void __launch_bounds__(kThreadsF)
    tc_featmap_kernel(const __grid_constant__ CUtensorMap tmap_x, int H, int N, int M,
                      const float* __restrict__ W1, const float* __restrict__ W2,
                      const float* __restrict__ rowscale, float scale,
                      __nv_bfloat16* __restrict__ phi, int* status)
{
    constexpr int P = NS ? 128 : 64;        // projection rows (= tensor memory columns) per group
    constexpr uint32_t NCOLS = G * P;        // 64, 128 or 256: a power of two
    constexpr uint32_t X0 = 0, W = 32768;    // two x tiles, then G x P frequency rows
    constexpr uint32_t WLO = W + G * P * 128; // their low parts
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sb = smem_u32(sm);
    __shared__ uint32_t tmem_base_sh;
    __shared__ __align__(8) uint64_t mbar, tma_bar[2];
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wg = warp >> 2, quad = warp & 3, t = 32 * quad + lane;
    const int nblk = (N + kC - 1) / kC, nchunk = (nblk + kBlocksPerCta - 1) / kBlocksPerCta;
    const int bh = blockIdx.x / nchunk, b0 = (blockIdx.x % nchunk) * kBlocksPerCta, h = bh % H;
    const int nb = min(kBlocksPerCta, nblk - b0);

    stage_freq_rows_split<NS, G, kThreadsF>(sb + W, sb + WLO, W1, W2, h, M, tid);  // once
    if (tid == 0) {
        mbar_init(&mbar, 1);
        mbar_init(&tma_bar[0], 1);
        mbar_init(&tma_bar[1], 1);
        abort_flag = 0;
        fence_mbar_init();
        mbar_arrive_expect_tx(&tma_bar[0], kTileBytes);
        tma_load_3d(sb + X0, &tmap_x, 0, b0 * kC, bh, &tma_bar[0]);
    }
    if (warp == 0) {
        tmem_alloc(&tmem_base_sh, NCOLS);
        tmem_relinquish();
    }
    fence_proxy_async();
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tm = tmem_base_sh;
    const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);
    constexpr uint32_t I_PROJ = idesc_bf16(128, P, 0, 0);

    bool ok = true;
    for (int r = 0; r < nb && ok; ++r) {
        const int blk = b0 + r, xb = r & 1;
        // the next tile into the other buffer (its projection finished last iteration)
        if (tid == 0 && r + 1 < nb) {
            mbar_arrive_expect_tx(&tma_bar[xb ^ 1], kTileBytes);
            tma_load_3d(sb + X0 + (xb ^ 1) * 16384, &tmap_x, 0, (blk + 1) * kC, bh,
                        &tma_bar[xb ^ 1]);
        }
        ok = bar_wait(&tma_bar[xb], (r >> 1) & 1, &abort_flag, status);
        ok = !__syncthreads_or(!ok);
        if (!ok) break;
        fence_after_sync();
        if (tid == 0) {
            const uint64_t dX = sdesc(sb + X0 + xb * 16384, 16, 1024);
            for (int g = 0; g < G; ++g) {
                const uint64_t dW = sdesc(sb + W + g * P * 128, 16, 1024);
                const uint64_t dWlo = sdesc(sb + WLO + g * P * 128, 16, 1024);
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_bf16(tm + g * P, dX + ((ks * 32) >> 4), dW + ((ks * 32) >> 4), I_PROJ,
                             ks > 0);
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_bf16(tm + g * P, dX + ((ks * 32) >> 4), dWlo + ((ks * 32) >> 4), I_PROJ,
                             1u);
            }
            mma_commit(&mbar);
        }
        ok = bar_wait(&mbar, r & 1, &abort_flag, status);
        ok = !__syncthreads_or(!ok);
        if (!ok) break;
        fence_after_sync();
        const int row = blk * kC + t;
        const bool valid = row < N;
        const float sc = scale * ((rowscale && valid) ? rowscale[(size_t)bh * N + row] : 1.f);
        __nv_bfloat16* out = phi + ((size_t)bh * N + (valid ? row : 0)) * 2 * M;
        for (int g = 0; g < G; ++g) {
            float a[32], w[32], m0, m1, m2 = 0.f, m3 = 0.f;  // m: max |x| per load
            const uint32_t col = tm_row + g * P + 32 * wg;
            tmem_ld16_maxabs(col, *reinterpret_cast<float(*)[16]>(&a[0]), m0);
            tmem_ld16_maxabs(col + 16, *reinterpret_cast<float(*)[16]>(&a[16]), m1);
            if (NS) {
                tmem_ld16_maxabs(col + 64, *reinterpret_cast<float(*)[16]>(&w[0]), m2);
                tmem_ld16_maxabs(col + 80, *reinterpret_cast<float(*)[16]>(&w[16]), m3);
            }
            tmem_wait_ld();
            const float mabs = fmaxf(fmaxf(m0, m1), fmaxf(m2, m3));
            if (NS)
                cos_w_args(a, w, mabs);  // w <- cos(w)
            else
                reduce_2pi_if_needed(a, mabs);
            uint32_t pc[16], ps[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                float s0, c0, s1, c1;
                __sincosf(a[2 * i], &s0, &c0);
                __sincosf(a[2 * i + 1], &s1, &c1);
                float k0 = sc, k1 = sc;
                if (NS) {
                    k0 *= w[2 * i];
                    k1 *= w[2 * i + 1];
                }
                pc[i] = pack_bf16(c0 * k0, c1 * k1);
                ps[i] = pack_bf16(s0 * k0, s1 * k1);
            }
            if (valid) {  // frequencies 64 g + 32 wg .. + 31: 64 contiguous bytes each
                uint4* dc = reinterpret_cast<uint4*>(out + 64 * g + 32 * wg);
                uint4* ds = reinterpret_cast<uint4*>(out + M + 64 * g + 32 * wg);
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    dc[j] = make_uint4(pc[4 * j], pc[4 * j + 1], pc[4 * j + 2], pc[4 * j + 3]);
                    ds[j] = make_uint4(ps[4 * j], ps[4 * j + 1], ps[4 * j + 2], ps[4 * j + 3]);
                }
            }
        }
        fence_before_sync();
        __syncthreads();  // tensor memory free for the next projection
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == 0) tmem_dealloc(tm, NCOLS);
}

template <bool NS, int G>
cudaError_t launch_typed(const Problem& p, const void* x, const float* W1, const float* W2,
                         const float* rowscale, void* phi, int* status, cudaStream_t s)
{
    CUtensorMap mx;
    const int BH = p.B * p.H;
    if (!make_act_map(&mx, x, BH, p.N)) return cudaErrorInvalidValue;
    constexpr int P = NS ? 128 : 64;
    const int smem = 32768 + 2 * G * P * 128 + 1024;
    auto kern = tc_featmap_kernel<NS, G>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const int nblk = (p.N + kC - 1) / kC;
    const long long blocks = (long long)BH * ((nblk + kBlocksPerCta - 1) / kBlocksPerCta);
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
    kern<<<(unsigned)blocks, kThreadsF, smem, s>>>(mx, p.H, p.N, p.M, W1, W2, rowscale,
                                                   1.0f / sqrtf((float)p.M),
                                                   (__nv_bfloat16*)phi, status);
    return cudaGetLastError();
}

}  // namespace

bool tc_featmap_supported(const Problem& p)
{
    return p.bf16 && p.d == 64 && (p.M == 64 || p.M == 128);
}

cudaError_t launch_tc_featmap(const Problem& p, const void* x, const float* W1, const float* W2,
                              const float* rowscale, void* phi, int* status, cudaStream_t s)
{
    if (p.nonstat)
        return p.M == 64 ? launch_typed<true, 1>(p, x, W1, W2, rowscale, phi, status, s)
                         : launch_typed<true, 2>(p, x, W1, W2, rowscale, phi, status, s);
    return p.M == 64 ? launch_typed<false, 1>(p, x, W1, W2, rowscale, phi, status, s)
                     : launch_typed<false, 2>(p, x, W1, W2, rowscale, phi, status, s);
}

}  // namespace flex
