// Attention-weight distillation loss on the tensor cores.
//
// The loss of the softmax-recovery experiments (the appendix's distillation setting): per
// query i the teacher distribution P_ij = softmax_j(q_i . k_j / sqrt(d)) and the kernel's
// normalised weights R_ij = A~_ij / D_i, A~_ij = phi~(q_i) . phi~(k_j), D_i = sum_l A~_il;
//   L = -(1/N) sum_i sum_j P_ij log R_ij     (j over all keys, or j <= i when causal).
// The query's prefactor and the feature scale cancel in R, so A~ uses phi(q) and the
// weighted key features w_j phi(k_j) (both written by a feature pass before this kernel).
// Entries with a non-positive R_ij count log(1e-6) (RFF estimates and row sums can be
// negative; the logarithm is undefined there).
//
// One CTA per (sequence, block of 128 queries), 256 threads: TMA loads the query tile and
// its features once, then per block of 128 keys the key tile and its features (the next
// block's load is issued once the MMAs have read the current one, so it overlaps the
// epilogue); thread 0 issues S = Q K^T (K = d = 64) into T_S and A = phi(Q) phi~(K)^T
// (K = 2M) into T_A; every thread then takes half of one query row's 128 columns and keeps
// online statistics in base 2: the running maximum m of the scores, Z = sum 2^(s-m), and
// for positive and negative A separately Z+- = sum 2^(s-m) and T+- = sum 2^(s-m) log2|A|,
// and D = sum A.  At the end the two halves merge and, by the sign of D,
//   L_i = -(ln2 T_sign - Z_sign ln|D| + (Z - Z_sign) ln 1e-6) / Z,
// which is the definition with the reading above applied.  Block sums of L_i go to
// partial slots, summed per sequence in a fixed order.  Every wait is bounded.
#include <algorithm>

#include "flex_internal.h"
#include "tc_common.cuh"
#include "tc_util.cuh"

namespace flex {
namespace {
using namespace tc;

constexpr int kC = 128;
constexpr int kThreadsA = 256;

template <int G2>  // 64-feature blocks of phi: 2M / 64
struct AwdCfg {
    static constexpr uint32_t Q = 0, K = 16384, PQ = 32768, PK = PQ + G2 * 16384;
    static constexpr uint32_t BYTES = PK + G2 * 16384;
    static constexpr uint32_t T_S = 0, T_A = 128;
    static_assert(BYTES + 1024 <= 232448, "shared memory budget");
};

__device__ __forceinline__ float ex2f(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float lg2f(float x)
{
    float y;
    asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

struct Stats {
    float m, z, zp, zn, tp, tn, den;
};

template <int G2>
__global__ void __launch_bounds__(kThreadsA, 1)
    tc_awd_kernel(const __grid_constant__ CUtensorMap tmap_q,
                  const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_pq,
                  const __grid_constant__ CUtensorMap tmap_pk, int N, int causal,
                  float score_scale, int nqb, float* __restrict__ part, int* status)
{
    using L = AwdCfg<G2>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sb = smem_u32(sm);
    __shared__ uint32_t tmem_base_sh;
    __shared__ __align__(8) uint64_t mbar, tma_bar;
    __shared__ volatile int abort_flag;
    __shared__ float merge[7][kC];
    __shared__ float wsum[kThreadsA / 32];

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wg = warp >> 2, quad = warp & 3, t = 32 * quad + lane;
    const int bh = blockIdx.x / nqb, qb = blockIdx.x % nqb;
    const int row = qb * kC + t;

    if (tid == 0) {
        mbar_init(&mbar, 1);
        mbar_init(&tma_bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0) {
        tmem_alloc(&tmem_base_sh, 256);
        tmem_relinquish();
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tm = tmem_base_sh;
    const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);
    uint32_t phase = 0, tma_phase = 0;
    auto adv = [](uint64_t dsc, uint32_t bytes) { return dsc + (bytes >> 4); };
    const uint64_t dQ = sdesc(sb + L::Q, 16, 1024), dK = sdesc(sb + L::K, 16, 1024);
    const uint64_t dPQ = sdesc(sb + L::PQ, 16, 1024), dPK = sdesc(sb + L::PK, 16, 1024);
    constexpr uint32_t I_KK128 = idesc_bf16(128, 128, 0, 0);

    Stats st = {-INFINITY, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    const int nkb = causal ? qb + 1 : (N + kC - 1) / kC;
    bool ok = true;

    // key tiles of block kb (one arrival per phase; the first also brings the query side)
    auto load_keys = [&](int kb) {
        mbar_arrive_expect_tx(&tma_bar, (1 + G2) * kTileBytes * (kb == 0 ? 2 : 1));
        if (kb == 0) {
            tma_load_3d(sb + L::Q, &tmap_q, 0, qb * kC, bh, &tma_bar);
            for (int g = 0; g < G2; ++g)
                tma_load_3d(sb + L::PQ + g * 16384, &tmap_pq, 64 * g, qb * kC, bh, &tma_bar);
        }
        tma_load_3d(sb + L::K, &tmap_k, 0, kb * kC, bh, &tma_bar);
        for (int g = 0; g < G2; ++g)
            tma_load_3d(sb + L::PK + g * 16384, &tmap_pk, 64 * g, kb * kC, bh, &tma_bar);
    };
    if (tid == 0) load_keys(0);
    for (int kb = 0; kb < nkb && ok; ++kb) {
        ok = bar_wait(&tma_bar, tma_phase, &abort_flag, status);
        tma_phase ^= 1;
        ok = !__syncthreads_or(!ok);
        if (!ok) break;
        fence_after_sync();
        if (tid == 0) {
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
                mma_bf16(tm + L::T_S, adv(dQ, ks * 32), adv(dK, ks * 32), I_KK128, ks > 0);
#pragma unroll
            for (int ks = 0; ks < 4 * G2; ++ks) {
                const uint32_t kofs = (ks >> 2) * 16384 + (ks & 3) * 32;
                mma_bf16(tm + L::T_A, adv(dPQ, kofs), adv(dPK, kofs), I_KK128, ks > 0);
            }
            mma_commit(&mbar);
        }
        ok = bar_wait(&mbar, phase, &abort_flag, status);
        phase ^= 1;
        ok = !__syncthreads_or(!ok);
        if (!ok) break;
        fence_after_sync();
        // the MMAs have read the key tiles: the next block's load overlaps this epilogue
        if (tid == 0 && kb + 1 < nkb) load_keys(kb + 1);
        // statistics over this thread's 64 columns, two rounds of 32; a block with no
        // masked key (not the ragged last one, not on the causal diagonal) takes the
        // unmasked path (rows past N are computed and discarded at the end)
        const bool full = (kb + 1) * kC <= N && (!causal || kb < qb);
#pragma unroll
        for (int b = 0; b < 2; ++b) {
            const uint32_t col = 64 * wg + 32 * b;
            float s[32], a[32];
            tmem_ld16(tm_row + L::T_S + col, *reinterpret_cast<float(*)[16]>(&s[0]));
            tmem_ld16(tm_row + L::T_S + col + 16, *reinterpret_cast<float(*)[16]>(&s[16]));
            tmem_ld16(tm_row + L::T_A + col, *reinterpret_cast<float(*)[16]>(&a[0]));
            tmem_ld16(tm_row + L::T_A + col + 16, *reinterpret_cast<float(*)[16]>(&a[16]));
            tmem_wait_ld();
            if (full) {  // no mask: every key of the block is valid for every row
                float bmax = s[0];
#pragma unroll
                for (int e = 1; e < 32; ++e) bmax = fmaxf(bmax, s[e]);
                bmax *= score_scale;  // > 0, so the maximum commutes with the scale
                if (bmax > st.m) {
                    const float f = ex2f(st.m - bmax);
                    st.z *= f; st.zp *= f; st.zn *= f; st.tp *= f; st.tn *= f;
                    st.m = bmax;
                }
                const float nm = -st.m;
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    const float p = ex2f(fmaf(s[e], score_scale, nm));
                    const float pl = p * lg2f(fabsf(a[e]));
                    st.z += p;
                    st.den += a[e];
                    if (a[e] > 0.f) { st.zp += p; st.tp += pl; }
                    if (a[e] < 0.f) { st.zn += p; st.tn += pl; }
                }
                continue;
            }
            const int j0 = kb * kC + (int)col;
            float bmax = -INFINITY;
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                const int j = j0 + e;
                const bool v = row < N && j < N && (!causal || j <= row);
                s[e] = v ? s[e] * score_scale : -INFINITY;
                bmax = fmaxf(bmax, s[e]);
            }
            if (bmax == -INFINITY) continue;  // no key of this round for this row
            if (bmax > st.m) {
                const float f = ex2f(st.m - bmax);  // 0 on the first valid round
                st.z *= f; st.zp *= f; st.zn *= f; st.tp *= f; st.tn *= f;
                st.m = bmax;
            }
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                if (s[e] == -INFINITY) continue;
                const float p = ex2f(s[e] - st.m);
                st.z += p;
                st.den += a[e];
                if (a[e] > 0.f) {
                    st.zp += p;
                    st.tp = fmaf(p, lg2f(a[e]), st.tp);
                } else if (a[e] < 0.f) {
                    st.zn += p;
                    st.tn = fmaf(p, lg2f(-a[e]), st.tn);
                }
            }
        }
        // tensor memory and the key tiles are free once every thread is here
        fence_before_sync();
        __syncthreads();
    }

    // merge the two halves of each row (wg 1 hands its statistics to wg 0)
    float lsum = 0.f;
    if (ok) {
        if (wg == 1) {
            merge[0][t] = st.m; merge[1][t] = st.z; merge[2][t] = st.zp; merge[3][t] = st.zn;
            merge[4][t] = st.tp; merge[5][t] = st.tn; merge[6][t] = st.den;
        }
        __syncthreads();
        if (wg == 0 && row < N) {
            const float m2 = merge[0][t], m = fmaxf(st.m, m2);
            const float f1 = st.m == -INFINITY ? 0.f : ex2f(st.m - m);
            const float f2 = m2 == -INFINITY ? 0.f : ex2f(m2 - m);
            const float z = st.z * f1 + merge[1][t] * f2;
            const float zp = st.zp * f1 + merge[2][t] * f2, zn = st.zn * f1 + merge[3][t] * f2;
            const float tp = st.tp * f1 + merge[4][t] * f2, tn = st.tn * f1 + merge[5][t] * f2;
            const float den = st.den + merge[6][t];
            constexpr float kLn2 = 0.69314718055994531f, kLnEps = -13.815510557964274f;  // ln 1e-6
            float li;
            if (den > 0.f)
                li = -(kLn2 * tp - zp * logf(den) + (z - zp) * kLnEps) / z;
            else if (den < 0.f)
                li = -(kLn2 * tn - zn * logf(-den) + (z - zn) * kLnEps) / z;
            else
                li = -kLnEps;
            lsum = li;
        }
    }
    // block sum in a fixed order
    for (int o = 16; o > 0; o >>= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
    if (lane == 0) wsum[warp] = lsum;
    __syncthreads();
    if (tid == 0) {
        float tot = 0.f;
        for (int w8 = 0; w8 < kThreadsA / 32; ++w8) tot += wsum[w8];
        part[blockIdx.x] = tot;
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == 0) tmem_dealloc(tm, 256);
}

__global__ void awd_reduce_kernel(int BH, int nqb, int N, const float* __restrict__ part,
                                  float* __restrict__ loss)
{
    for (int u = blockIdx.x * blockDim.x + threadIdx.x; u < BH; u += gridDim.x * blockDim.x) {
        float s = 0.f;
        for (int b = 0; b < nqb; ++b) s += part[(size_t)u * nqb + b];  // fixed order
        loss[u] = s / (float)N;
    }
}

template <int G2>
cudaError_t launch_typed(const Problem& p, const void* q, const void* k, const void* pq,
                         const void* pk, float* part, float* loss, int* status, cudaStream_t s)
{
    const int BH = p.B * p.H, nqb = (p.N + kC - 1) / kC;
    CUtensorMap mq, mk, mpq, mpk;
    if (!make_act_map(&mq, q, BH, p.N) || !make_act_map(&mk, k, BH, p.N) ||
        !make_feat_map(&mpq, pq, BH, p.N, 2 * p.M) || !make_feat_map(&mpk, pk, BH, p.N, 2 * p.M))
        return cudaErrorInvalidValue;
    const int smem = (int)AwdCfg<G2>::BYTES + 1024;
    auto kern = tc_awd_kernel<G2>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const float score_scale = 1.4426950408889634f / sqrtf((float)p.d);  // log2(e) / sqrt(d)
    kern<<<BH * nqb, kThreadsA, smem, s>>>(mq, mk, mpq, mpk, p.N, p.causal, score_scale, nqb,
                                           part, status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    awd_reduce_kernel<<<(BH + 255) / 256, 256, 0, s>>>(BH, nqb, p.N, part, loss);
    return cudaGetLastError();
}

}  // namespace

bool tc_awd_supported(const Problem& p)
{
    return p.bf16 && p.d == 64 && (p.M == 64 || p.M == 128);
}

size_t tc_awd_part_floats(const Problem& p)
{
    return (size_t)p.B * p.H * ((p.N + kC - 1) / kC);
}

cudaError_t launch_tc_awd(const Problem& p, const void* q, const void* k, const void* pq,
                          const void* pk, float* part, float* loss, int* status, cudaStream_t s)
{
    return p.M == 64 ? launch_typed<2>(p, q, k, pq, pk, part, loss, status, s)
                     : launch_typed<4>(p, q, k, pq, pk, part, loss, status, s);
}

}  // namespace flex
