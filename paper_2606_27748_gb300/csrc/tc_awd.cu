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
// partial slots, summed per sequence in a fixed order.  Every wait is bounded.  For the
// gradient the same kernel also writes each row's statistics (below).
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
                  float score_scale, int nqb, float* __restrict__ part,
                  float4* __restrict__ rowstat, int* status)
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
            if (rowstat) {  // what the gradient needs of this row (see the gradient kernel)
                const float sg = den > 0.f ? 1.f : (den < 0.f ? -1.f : 0.f);
                const float zs = den > 0.f ? zp : zn;
                const float e = sg != 0.f ? (zs / z) / den : 0.f;
                rowstat[(size_t)bh * N + row] = make_float4(m + log2f(z), sg, e, 0.f);
            }
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

// ---- gradient with respect to the kernel's parameters ------------------------------------
//
// The distillation trains only the feature map, so the gradient is taken with respect to
// W1, W2 and tau.  With the row statistics of the loss kernel (l_i = log2 of the softmax
// normaliser in the scaled base-2 scores, the sign of D_i, e_i = c_i / D_i where c_i is the
// teacher mass on the entries with R_ij > 0) and sigma = -dloss / N:
//   dL/dA~_ij = sigma G_ij,   G_ij = [A~_ij sign(D_i) > 0] P_ij / A~_ij - e_i   (j in row i)
//   dphi(q_i) = sigma sum_j G_ij phi~(k_j),   dphi~(k_j) = sigma sum_i G_ij phi(q_i).
// A sequence's query side holds blocks of 128 queries and streams the key blocks; its key
// side holds blocks of 128 keys and streams the query blocks; each side's held blocks are
// split over `hsplit` CTAs.  Per streamed block thread 0 issues S = X_own X_other^T and
// A = Phi_own Phi_other^T into tensor memory; 16 warps (four per lane quadrant, each on 32
// of the 128 columns) turn their part of the rows into G (two SFU operations per entry:
// ex2 and a divide), write it as bf16 in place over the columns they read, and G Phi_other
// (A operand in tensor memory, features MN-major) accumulates into T_D.  With M = 64 the
// streamed tiles are double-buffered: the next block's load is issued as soon as the
// current one has landed.  Then, per group of 64 frequencies, the chain rule through the
// feature map runs on the tensor cores: the projection X_own W'^T is recomputed, the
// epilogue forms da (du | dw for Flexformer_n) from T_D, and dW' += da^T X_own.  The rows of
// dW' are added into this CTA's slot; a reduction sums the slots over the sides, the batch
// and the splits in a fixed order, so the result does not depend on scheduling.  On the
// key side, with the prefactor, the chain rule takes dphi(k_j) = w_j dphi~(k_j) and dtau
// gains -(phi~(k_j) . dphi~(k_j)) |k_j|^2 exp(-tau).  Every wait is bounded.
constexpr int kThreadsG = 512;

template <int G2>
struct AwdBwCfg {
    static constexpr int STAGES = G2 == 2 ? 2 : 1;          // streamed tiles in flight
    static constexpr uint32_t XO = 0, PO = 16384, ST0 = PO + G2 * 16384;
    static constexpr uint32_t STAGE_BYTES = (1 + G2) * 16384;  // x tile, then features
    static constexpr uint32_t WG = ST0 + STAGES * STAGE_BYTES;  // W' rows of every group
    static constexpr uint32_t BYTES = WG + (G2 / 2) * 16384;   // (at most 16 KB a group)
    static constexpr uint32_t DA = ST0 + 16384;  // after the streamed blocks: da [du | dw]
    static constexpr uint32_t T_S = 0, T_A = 128, T_D = 256;
    static_assert(G2 >= 2 && BYTES + 1024 <= 232448, "shared memory budget");
};

template <int G2, bool NS, bool KW>
__global__ void __launch_bounds__(kThreadsG, 1)
    tc_awd_bwd_kernel(const __grid_constant__ CUtensorMap tmap_q,
                      const __grid_constant__ CUtensorMap tmap_k,
                      const __grid_constant__ CUtensorMap tmap_pq,
                      const __grid_constant__ CUtensorMap tmap_pk, int BH, int H, int N, int M,
                      int causal, int hsplit, float score_scale,
                      const float4* __restrict__ rowstat, const float* __restrict__ dloss,
                      const float* __restrict__ W1, const float* __restrict__ W2,
                      const float* __restrict__ kw, const float* __restrict__ tau,
                      float* __restrict__ slots, float* __restrict__ dtau_part, int* status)
{
    using L = AwdBwCfg<G2>;
    constexpr int P = NS ? 128 : 64;  // projection rows per group of 64 frequencies
    constexpr int G = G2 / 2;
    constexpr int S = L::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sb = smem_u32(sm);
    __shared__ uint32_t tmem_base_sh;
    __shared__ __align__(8) uint64_t mbar, tma_bar[S];
    __shared__ volatile int abort_flag;
    __shared__ float4 ostat[kC];  // key side: statistics of the streamed query rows
    __shared__ float wsum[kThreadsG / 32];

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int qd = warp >> 2, quad = warp & 3, t = 32 * quad + lane;  // qd: column quarter
    const int seq = (int)blockIdx.x / hsplit, split = (int)blockIdx.x % hsplit;
    const bool kside = seq >= BH;
    const int bh = seq % BH, h = bh % H;
    const CUtensorMap* x_own = kside ? &tmap_k : &tmap_q;
    const CUtensorMap* x_oth = kside ? &tmap_q : &tmap_k;
    const CUtensorMap* f_own = kside ? &tmap_pk : &tmap_pq;
    const CUtensorMap* f_oth = kside ? &tmap_pq : &tmap_pk;
    const int nblk = (N + kC - 1) / kC;
    const int hb0 = split * nblk / hsplit, hb1 = (split + 1) * nblk / hsplit;
    const float sigma = -dloss[bh] / (float)N;
    const float itau = KW ? expf(-tau[h]) : 0.f;
    const float cM = rsqrtf((float)M);
    float dtau_acc = 0.f;

    if (tid == 0) {
        mbar_init(&mbar, 1);
        for (int s = 0; s < S; ++s) mbar_init(&tma_bar[s], 1);
        abort_flag = 0;
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
    const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);
    uint32_t phase = 0, tph = 0;  // tph: bit st = parity of stage st's barrier
    auto adv = [](uint64_t dsc, uint32_t bytes) { return dsc + (bytes >> 4); };
    auto xt = [](int st) { return L::ST0 + (uint32_t)st * L::STAGE_BYTES; };
    const uint64_t dXO = sdesc(sb + L::XO, 16, 1024), dPO = sdesc(sb + L::PO, 16, 1024);
    const uint64_t dDAmn = sdesc(sb + L::DA, 16384, 1024), dXOmn = sdesc(sb + L::XO, 16384, 1024);
    constexpr uint32_t I_KK128 = idesc_bf16(128, 128, 0, 0);
    constexpr uint32_t I_DPHI = idesc_bf16(128, 64 * G2, 0, 1);  // N = 2M features
    constexpr uint32_t I_PROJ = idesc_bf16(128, P, 0, 0);
    constexpr uint32_t I_DW = idesc_bf16(128, 64, 1, 1);

    auto handoff = [&]() {
        fence_proxy_async();
        fence_before_sync();
        __syncthreads();
    };
    auto commit_wait = [&]() -> bool {  // thread 0 has issued MMAs: commit, all wait
        if (tid == 0) mma_commit(&mbar);
        bool ok_ = bar_wait(&mbar, phase, &abort_flag, status);
        phase ^= 1;
        ok_ = !__syncthreads_or(!ok_);
        fence_after_sync();
        return ok_;
    };
    // streamed block ot into stage st (and first the held block ob): one arrival per phase
    auto load = [&](int ob, int ot, int st, bool own_too) {
        mbar_arrive_expect_tx(&tma_bar[st], (1 + G2) * kTileBytes * (own_too ? 2 : 1));
        if (own_too) {
            tma_load_3d(sb + L::XO, x_own, 0, ob * kC, bh, &tma_bar[st]);
            for (int g = 0; g < G2; ++g)
                tma_load_3d(sb + L::PO + g * 16384, f_own, 64 * g, ob * kC, bh, &tma_bar[st]);
        }
        tma_load_3d(sb + xt(st), x_oth, 0, ot * kC, bh, &tma_bar[st]);
        for (int g = 0; g < G2; ++g)
            tma_load_3d(sb + xt(st) + 16384 + g * 16384, f_oth, 64 * g, ot * kC, bh,
                        &tma_bar[st]);
    };
    // streamed blocks of held block ob: causal queries see keys j <= i
    auto first_other = [&](int ob) { return (kside && causal) ? ob : 0; };
    auto last_other = [&](int ob) { return (!kside && causal) ? ob : nblk - 1; };

    bool ok = true;
    if (tid == 0) load(hb0, first_other(hb0), 0, true);
    // this head's W' rows, all groups, once (overlaps the first load; made visible to the
    // tensor cores by the fence here and the barrier at the first wait)
    stage_freq_rows<NS, G, kThreadsG>(sb + L::WG, W1, W2, h, M, tid);
    fence_proxy_async();
    for (int ob = hb0; ob < hb1 && ok; ++ob) {
        const int own_row = ob * kC + t;
        const bool own_valid = own_row < N;
        float4 qs = make_float4(0.f, 0.f, 0.f, 0.f);
        if (!kside && own_valid) qs = rowstat[(size_t)bh * N + own_row];
        const int o0 = first_other(ob), o1 = last_other(ob);
        for (int ot = o0; ot <= o1; ++ot) {
            const int st = S == 2 ? (ot - o0) & 1 : 0;
            if (kside && tid < kC) {
                const int r = ot * kC + tid;
                ostat[tid] = r < N ? rowstat[(size_t)bh * N + r] : make_float4(0.f, 0.f, 0.f, 0.f);
            }
            ok = bar_wait(&tma_bar[st], (tph >> st) & 1u, &abort_flag, status);
            tph ^= 1u << st;
            ok = !__syncthreads_or(!ok);
            if (!ok) break;
            fence_after_sync();
            if (tid == 0) {
                // the other stage was last read by the previous block's MMAs, now complete
                if (S == 2 && ot < o1) load(ob, ot + 1, st ^ 1, false);
                const uint64_t dXT = sdesc(sb + xt(st), 16, 1024);
                const uint64_t dPT = sdesc(sb + xt(st) + 16384, 16, 1024);
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_bf16(tm + L::T_S, adv(dXO, ks * 32), adv(dXT, ks * 32), I_KK128, ks > 0);
#pragma unroll
                for (int ks = 0; ks < 4 * G2; ++ks) {
                    const uint32_t kofs = (ks >> 2) * 16384 + (ks & 3) * 32;
                    mma_bf16(tm + L::T_A, adv(dPO, kofs), adv(dPT, kofs), I_KK128, ks > 0);
                }
            }
            if (!(ok = commit_wait())) break;
            // G over this thread's 32 columns (two rounds of 16), bf16 in place over A in
            // the first 16 of them; a block with no masked entry skips the mask tests
            const bool full = (ot + 1) * kC <= N && (ob + 1) * kC <= N &&
                              (!causal || (kside ? ot > ob : ot < ob));
#pragma unroll
            for (int b = 0; b < 2; ++b) {
                const uint32_t col = 32 * qd + 16 * b;
                float sv[16], av[16];
                tmem_ld16(tm_row + L::T_S + col, sv);
                tmem_ld16(tm_row + L::T_A + col, av);
                tmem_wait_ld();
                uint32_t pk[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    float gv[2];
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const int c = (int)col + 2 * i + e;
                        const float4 sts = kside ? ostat[c] : qs;
                        const float a = av[2 * i + e];
                        const float p = ex2f(fmaf(sv[2 * i + e], score_scale, -sts.x));
                        const float g = (a * sts.y > 0.f ? __fdividef(p, a) : 0.f) - sts.z;
                        if (full) {
                            gv[e] = g;
                        } else {
                            const int orow = ot * kC + c;
                            const int qi = kside ? orow : own_row, kj = kside ? own_row : orow;
                            gv[e] = (own_valid && orow < N && (!causal || kj <= qi)) ? g : 0.f;
                        }
                    }
                    pk[i] = pack_bf16(gv[0], gv[1]);
                }
                tmem_st8(tm_row + L::T_A + 32 * qd + 8 * b, pk);
            }
            tmem_wait_st();
            handoff();
            if (tid == 0) {
                fence_after_sync();
                const uint64_t dPTmn = sdesc(sb + xt(st) + 16384, 16384, 1024);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)  // K = streamed rows 16 ks .. 16 ks + 15
                    mma_bf16_tmem_a(tm + L::T_D, tm + L::T_A + 32 * (ks >> 1) + 8 * (ks & 1),
                                    adv(dPTmn, ks * 2048), I_DPHI, (ot > o0 || ks > 0) ? 1u : 0u);
            }
            if (!(ok = commit_wait())) break;
            if (S == 1 && tid == 0 && ot < o1) load(ob, ot + 1, 0, false);
        }
        if (!ok) break;

        // chain rule through the feature map, one group of 64 frequencies at a time
        const float wk = (KW && kside && own_valid) ? kw[(size_t)bh * N + own_row] : 1.f;
        const float scl = sigma * wk;  // dphi(x) = scl T_D (key side: dphi = w dphi~)
        float sdot = 0.f;              // key side: phi(k) . T_D over this thread's features
        float kk = 0.f;                // key side: |k_j|^2 from the held tile (read before
        if (KW && kside) {             // the group loop: the next block's load reuses it)
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const uint4 k4 = *reinterpret_cast<const uint4*>(sm + L::XO + swz128(t, 8 * j));
                const uint32_t kw4[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float k0 = __uint_as_float(kw4[e] << 16);
                    const float k1 = __uint_as_float(kw4[e] & 0xFFFF0000u);
                    kk = fmaf(k0, k0, fmaf(k1, k1, kk));
                }
            }
        }
        for (int g = 0; g < G && ok; ++g) {
            if (tid == 0) {
                fence_after_sync();  // after the previous group's barrier
                const uint64_t dWg = sdesc(sb + L::WG + (uint32_t)g * P * 128, 16, 1024);
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_bf16(tm + L::T_S, adv(dXO, ks * 32), adv(dWg, ks * 32), I_PROJ, ks > 0);
            }
            if (!(ok = commit_wait())) break;
            // this thread's 16 frequencies of the group: 64 g + 16 qd + [0, 16)
            float dc[16], ds[16], u[16], w[16];
            tmem_ld16(tm_row + L::T_D + 64 * g + 16 * qd, dc);
            tmem_ld16(tm_row + L::T_D + M + 64 * g + 16 * qd, ds);
            float mu, mw = 0.f;  // max |x| per load
            tmem_ld16_maxabs(tm_row + L::T_S + 16 * qd, u, mu);
            if (NS) tmem_ld16_maxabs(tm_row + L::T_S + 64 + 16 * qd, w, mw);
            tmem_wait_ld();
            if (NS)
                reduce_2pi_if_needed(u, w, fmaxf(mu, mw));
            else
                reduce_2pi_if_needed(u, mu);
            uint32_t o1[8], o2[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                float r1[2], r2[2];
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int f = 2 * i + e;
                    float su, cu;
                    __sincosf(u[f], &su, &cu);
                    float cw = 1.f, sw = 0.f;
                    if (NS) __sincosf(w[f], &sw, &cw);
                    const float dpc = scl * dc[f], dps = scl * ds[f];
                    r1[e] = cM * cw * (-su * dpc + cu * dps);
                    r2[e] = NS ? -cM * sw * (cu * dpc + su * dps) : 0.f;
                    if (KW) sdot = fmaf(cu * cw, dc[f], fmaf(su * cw, ds[f], sdot));
                    if (!own_valid) r1[e] = r2[e] = 0.f;
                }
                o1[i] = pack_bf16(r1[0], r1[1]);
                o2[i] = pack_bf16(r2[0], r2[1]);
            }
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                const uint32_t off = swz128(t, (2 * qd + j) * 8);
                st_shared_v4(sb + L::DA + off, o1[4 * j], o1[4 * j + 1], o1[4 * j + 2], o1[4 * j + 3]);
                st_shared_v4(sb + L::DA + 16384 + off, o2[4 * j], o2[4 * j + 1], o2[4 * j + 2],
                             o2[4 * j + 3]);
            }
            handoff();
            if (tid == 0) {
                fence_after_sync();
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_bf16(tm + L::T_A, adv(dDAmn, ks * 2048), adv(dXOmn, ks * 2048), I_DW, ks > 0);
            }
            if (!(ok = commit_wait())) break;
            // rows of dW' (lane = projection row), this thread's 16 columns, into the slot
            float v[16];
            tmem_ld16(tm_row + L::T_A + 16 * qd, v);
            tmem_wait_ld();
            float4* dst = reinterpret_cast<float4*>(
                slots + (((size_t)blockIdx.x * G + g) * 128 + t) * 64 + 16 * qd);
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const float4 old = ob == hb0 ? make_float4(0.f, 0.f, 0.f, 0.f) : dst[j];
                dst[j] = make_float4(old.x + v[4 * j], old.y + v[4 * j + 1], old.z + v[4 * j + 2],
                                     old.w + v[4 * j + 3]);
            }
            // tensor memory, the W' rows and the da tiles are free once every thread is here
            fence_before_sync();
            __syncthreads();
        }
        if (!ok) break;
        if (KW && kside && own_valid)  // s_j = phi~(k_j) . dphi~(k_j) = w cM sigma sdot
            dtau_acc -= wk * cM * sigma * sdot * kk * itau;
        if (tid == 0 && ob + 1 < hb1) load(ob + 1, first_other(ob + 1), 0, true);
    }

    // dtau partial of this CTA, summed in a fixed order
    float dsum = dtau_acc;
    for (int o = 16; o > 0; o >>= 1) dsum += __shfl_xor_sync(0xffffffffu, dsum, o);
    if (lane == 0) wsum[warp] = dsum;
    __syncthreads();
    if (tid == 0) {
        float tot = 0.f;
        for (int w8 = 0; w8 < kThreadsG / 32; ++w8) tot += wsum[w8];
        dtau_part[blockIdx.x] = tot;
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == 0) tmem_dealloc(tm, 512);
}

// dW1, dW2 [H][M][64] and dtau [H] from the slots [2 sides][B*H][hsplit][G][128 rows][64].
// One block of 512 threads per (head, frequency): column c = tid % 64, lane = tid / 64 sums
// the slots s = lane, lane + 8, ... (s in (side, batch entry, split) order), eight loads in
// flight; the eight lane sums are then added in lane order, so the order is fixed.  For
// Flexformer_n rows 0-63 of a group are dU, rows 64-127 dV (U = (W1+W2)/2, V = (W1-W2)/2),
// so dW1 = (dU+dV)/2, dW2 = (dU-dV)/2.
constexpr int kReduceLanes = 8;
__global__ void __launch_bounds__(64 * kReduceLanes)
    awd_dw_reduce_kernel(int B, int H, int M, int nonstat, int hsplit,
                         const float* __restrict__ slots, const float* __restrict__ dtau_part,
                         float* __restrict__ dW1, float* __restrict__ dW2,
                         float* __restrict__ dtau)
{
    __shared__ float part[2][kReduceLanes][64];
    const int BH = B * H, G = M / 64, per_side = B * hsplit, nslot = 2 * per_side;
    const size_t slot_floats = (size_t)G * 128 * 64;
    const int c = threadIdx.x % 64, lane = threadIdx.x / 64;
    const int f = blockIdx.x % M, h = blockIdx.x / M;
    const float* base = slots + ((size_t)(f / 64) * 128 + f % 64) * 64 + c;
    float su = 0.f, sv = 0.f;
    for (int s0 = lane; s0 < nslot; s0 += 8 * kReduceLanes) {
        float a[8], bq[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int s = s0 + e * kReduceLanes;
            a[e] = bq[e] = 0.f;
            if (s < nslot) {
                const int side = s / per_side, rem = s % per_side;
                const size_t cta = (size_t)(side * BH + (rem / hsplit) * H + h) * hsplit +
                                   rem % hsplit;
                a[e] = base[cta * slot_floats];
                if (nonstat) bq[e] = base[cta * slot_floats + 64 * 64];
            }
        }
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            su += a[e];
            sv += bq[e];
        }
    }
    part[0][lane][c] = su;
    part[1][lane][c] = sv;
    __syncthreads();
    if (lane == 0) {
        float tu = 0.f, tv = 0.f;
        for (int l = 0; l < kReduceLanes; ++l) {
            tu += part[0][l][c];
            tv += part[1][l][c];
        }
        const size_t idx = ((size_t)h * M + f) * 64 + c;
        if (nonstat) {
            dW1[idx] = 0.5f * (tu + tv);
            dW2[idx] = 0.5f * (tu - tv);
        } else {
            dW1[idx] = tu;
        }
    }
    if (dtau && blockIdx.x == 0)
        for (int hh = threadIdx.x; hh < H; hh += blockDim.x) {
            float sd = 0.f;
            for (int b = 0; b < B; ++b)
                for (int r = 0; r < hsplit; ++r)  // key side
                    sd += dtau_part[(size_t)(BH + b * H + hh) * hsplit + r];
            dtau[hh] = sd;
        }
}

template <int G2>
cudaError_t launch_typed(const Problem& p, const void* q, const void* k, const void* pq,
                         const void* pk, float* part, float* loss, float4* rowstat, int* status,
                         cudaStream_t s)
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
                                           part, rowstat, status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (!loss) return cudaSuccess;
    awd_reduce_kernel<<<(BH + 255) / 256, 256, 0, s>>>(BH, nqb, p.N, part, loss);
    return cudaGetLastError();
}

// CTAs per (side, sequence) of the gradient kernel: held blocks are split until the grid
// covers the GPU about four times over (whole blocks per CTA).
int awd_hsplit(const Problem& p)
{
    const int nblk = (p.N + kC - 1) / kC;
    int hs = 1;
    while (hs * 2 <= nblk && 2LL * p.B * p.H * hs < 4LL * 152) hs *= 2;
    return hs;
}

template <int G2, bool NS, bool KW>
cudaError_t launch_bwd_typed(const Problem& p, const void* q, const void* k, const void* pq,
                             const void* pk, const float* W1, const float* W2, const float* kw,
                             const float* tau, const float* dloss, const float4* rowstat,
                             float* slots, float* dtau_part, float* dW1, float* dW2, float* dtau,
                             int* status, cudaStream_t s)
{
    const int BH = p.B * p.H;
    CUtensorMap mq, mk, mpq, mpk;
    if (!make_act_map(&mq, q, BH, p.N) || !make_act_map(&mk, k, BH, p.N) ||
        !make_feat_map(&mpq, pq, BH, p.N, 2 * p.M) || !make_feat_map(&mpk, pk, BH, p.N, 2 * p.M))
        return cudaErrorInvalidValue;
    const int smem = (int)AwdBwCfg<G2>::BYTES + 1024;
    auto kern = tc_awd_bwd_kernel<G2, NS, KW>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const float score_scale = 1.4426950408889634f / sqrtf((float)p.d);
    const int hs = awd_hsplit(p);
    kern<<<2 * BH * hs, kThreadsG, smem, s>>>(mq, mk, mpq, mpk, BH, p.H, p.N, p.M, p.causal, hs,
                                              score_scale, rowstat, dloss, W1, W2, kw, tau, slots,
                                              dtau_part, status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    awd_dw_reduce_kernel<<<p.H * p.M, 64 * kReduceLanes, 0, s>>>(
        p.B, p.H, p.M, p.nonstat, hs, slots, dtau_part, dW1, dW2, tau ? dtau : nullptr);
    return cudaGetLastError();
}

template <int G2>
cudaError_t launch_bwd_g2(const Problem& p, const void* q, const void* k, const void* pq,
                          const void* pk, const float* W1, const float* W2, const float* kw,
                          const float* tau, const float* dloss, const float4* rowstat,
                          float* slots, float* dtau_part, float* dW1, float* dW2, float* dtau,
                          int* status, cudaStream_t s)
{
    if (p.nonstat)
        return tau ? launch_bwd_typed<G2, true, true>(p, q, k, pq, pk, W1, W2, kw, tau, dloss,
                                                      rowstat, slots, dtau_part, dW1, dW2, dtau,
                                                      status, s)
                   : launch_bwd_typed<G2, true, false>(p, q, k, pq, pk, W1, W2, kw, tau, dloss,
                                                       rowstat, slots, dtau_part, dW1, dW2, dtau,
                                                       status, s);
    return tau ? launch_bwd_typed<G2, false, true>(p, q, k, pq, pk, W1, W2, kw, tau, dloss,
                                                   rowstat, slots, dtau_part, dW1, dW2, dtau,
                                                   status, s)
               : launch_bwd_typed<G2, false, false>(p, q, k, pq, pk, W1, W2, kw, tau, dloss,
                                                    rowstat, slots, dtau_part, dW1, dW2, dtau,
                                                    status, s);
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

size_t tc_awd_slot_floats(const Problem& p)
{
    return (size_t)2 * p.B * p.H * awd_hsplit(p) * (p.M / 64) * 128 * 64;
}

cudaError_t launch_tc_awd(const Problem& p, const void* q, const void* k, const void* pq,
                          const void* pk, float* part, float* loss, int* status, cudaStream_t s)
{
    return p.M == 64 ? launch_typed<2>(p, q, k, pq, pk, part, loss, nullptr, status, s)
                     : launch_typed<4>(p, q, k, pq, pk, part, loss, nullptr, status, s);
}

cudaError_t launch_tc_awd_bwd(const Problem& p, const void* q, const void* k, const void* pq,
                              const void* pk, const float* W1, const float* W2, const float* kw,
                              const float* tau, const float* dloss, float* part, float* loss,
                              float4* rowstat, float* slots, float* dtau_part, float* dW1,
                              float* dW2, float* dtau, int* status, cudaStream_t s)
{
    cudaError_t e = p.M == 64 ? launch_typed<2>(p, q, k, pq, pk, part, loss, rowstat, status, s)
                              : launch_typed<4>(p, q, k, pq, pk, part, loss, rowstat, status, s);
    if (e != cudaSuccess) return e;
    return p.M == 64 ? launch_bwd_g2<2>(p, q, k, pq, pk, W1, W2, kw, tau, dloss, rowstat, slots,
                                        dtau_part, dW1, dW2, dtau, status, s)
                     : launch_bwd_g2<4>(p, q, k, pq, pk, W1, W2, kw, tau, dloss, rowstat, slots,
                                        dtau_part, dW1, dW2, dtau, status, s);
}

}  // namespace flex
