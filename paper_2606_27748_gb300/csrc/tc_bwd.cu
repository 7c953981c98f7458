// Backward of RFF linear attention on the tensor cores (tcgen05).
//
// Gradient of L = sum(dout * out) for Eq. (linear att).  With unscaled features phi'
// (the M^{-1/2} cancels), den' = M den, g_i = dout_i / den'_i, c_i = -(dout_i . out_i)/den'_i:
//   dA_ij    = g_i . v_j + c_i                      (j <= i when causal)
//   dphi(q_i) = sum_j dA_ij phi(k_j)   = [intra-chunk] + S_i g_i + c_i z_i
//   dphi(k_j) = sum_i dA_ij phi(q_i)   = [intra-chunk] + R_j v_j + r_j
//   dv_j      = sum_i A_ij g_i         = [intra-chunk] + R_j^T phi(k_j)
// with S = sum phi(k) v^T, z = sum phi(k) (forward running sums) and R = sum phi(q) g^T,
// r = sum c phi(q) (reverse running sums), then through the feature map (Eq. phi_n /
// phi_non) by the chain rule: dx = da W, dW += da^T x.
//
// Every term splits over feature groups (64 frequencies = 128 features), and A enters dv
// linearly, so one CTA handles one (sequence, group) pair and the group results are summed.
// With two groups (M = 128) the two CTAs of a (pass, sequence) form a cluster: each chunk,
// CTA r finishes rows 64r..64r+63 of dq (pass F) or dk and dv (pass R): it sends its
// fp32 partial rows of the other half to the partner (staged in its own shared memory, one
// bulk copy into a region the partner has declared free), adds the partner's partial to its
// own rows and stores bf16.  dW goes through per-(pass, sequence, group) partials reduced
// over the batch in a fixed order.  Pass F runs the chunks forward (dq and the q part of
// dW, state S, z), pass R runs them backward (dk, dv and the k part of dW, state R, r); the
// two are independent and run as the two halves of one grid, pass R (the longer) first.
//
// Norm prefactor (Sec. 3.2, optional): with key weights w_j = exp(|k_j|^2 exp(-tau)) (kw,
// one pass over k before this kernel), phi(k) is stored weighted, so S, z, A and dv come
// out weighted and T_D holds the gradient with respect to the weighted features.  In pass
// R the chain rule then needs dphi(k) = w dphi~(k) (the stationary feature tile already
// carries w; the nonstationary recomputation multiplies by it), s_j = phi~(k_j).dphi~(k_j)
// adds 2 exp(-tau) s_j k_j to dk_j (folded into the same row adds) and -ln(w_j) s_j to
// dtau (per-CTA slots, reduced with dW in a fixed order).
//
// Phases run in order inside a CTA: all 256 threads load, compute features and run the
// CUDA-core epilogues; thread 0 issues the MMAs; one mbarrier tracks their completion
// (bounded waits).  The next chunk's q / k / v / dout / out tiles are loaded as soon as
// the region each one occupies is free, and each exchange is sent at once and finished
// later (dq and dk rows at the start of the next chunk, dv before the projection
// backward), so the copies and the partner's progress overlap this CTA's work.
//
// Exchange regions (staging -> the partner's receive region; each free when it is used):
//   causal   pass F  dq: PQ -> PK        pass R  dv: PQ -> DA2, dk: PQ+16K -> GT
//   kGrad    pass F  dq: K  -> PK        pass R  dv: Q  -> DO,  dk: DA2 -> O
//
// Tensor memory (512 columns): [0,128) projection, [128,256) A / dA (bf16 in place) then
// dx (0-63) and the chunk's dW (64-127), [256,384) dphi, [384,464) S|z or R|r.
#include <algorithm>

#include "flex_internal.h"
#include "tc_common.cuh"
#include "tc_util.cuh"

namespace flex {
namespace {
using namespace tc;

constexpr int kC = 128;
constexpr int kThreadsB = 256;
constexpr uint32_t kXBytes = 64 * 64 * 4;  // one exchanged half: 64 rows x 64 fp32
enum { kPassF = 0, kPassR = 1 };
// kCausal: the chunked scans of the causal gradient.  Non-causal (every key for every query):
// kState sums partial states over a range of chunks (pass F: [S | z] = sum phi(k) [v | 1],
// pass R: [R | r] = sum phi(q) [g | c]); kGrad starts from their totals and needs no scan:
// pass F dphi(q) = S g + c z, pass R dphi(k) = R v + r and dv = R^T phi(k).
enum { kCausal = 0, kState = 1, kGrad = 2 };

template <bool NS>
struct BwCfg {
    static constexpr int P = NS ? 128 : 64;  // projection rows (and dW rows) per group
    // shared memory (bytes).  Pass R keeps bf16(dA) in [Q | DA2] and bf16(A) in [DO | O].
    static constexpr uint32_t Q = 0, DA2 = 16384, K = 32768, V = 49152, DO = 65536, O = 81920;
    static constexpr uint32_t GT = 98304;     // g tile [token][dcol], bf16
    static constexpr uint32_t C16 = 114688;   // K-major [16][128 tokens]: ones (F) / c (R)
    static constexpr uint32_t W = 118784;     // this group's projection rows
    static constexpr uint32_t PQ = 135168, PK = 167936;  // features (then da in place)
    static constexpr uint32_t SN = 200704;    // state snapshot [feature][64 dcol], bf16
    static constexpr uint32_t ZR = 217088;    // z or r [128] fp32
    static constexpr uint32_t CROW = 217600;  // c_t [128] fp32
    static constexpr uint32_t SPART = 218112; // prefactor: s_t partials [2 warpgroups][128]
    static constexpr uint32_t BYTES = 219136;
    static constexpr uint32_t T_P = 0, T_A = 128, T_D = 256, T_S = 384;
    static_assert(BYTES + 1024 <= 232448, "shared memory budget");
};


__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// KW: key weights of the norm prefactor given (compile-time; the plain kernel is unchanged);
// CS: CTAs per cluster = frequency groups (1 or 2; 1 for kState, which exchanges nothing);
// MODE: kCausal, kState or kGrad
template <bool NS, bool KW, int CS, int MODE>
__global__ void __launch_bounds__(kThreadsB, 1)
    tc_bwd_kernel(const __grid_constant__ CUtensorMap tmap_q,
                  const __grid_constant__ CUtensorMap tmap_k,
                  const __grid_constant__ CUtensorMap tmap_v,
                  const __grid_constant__ CUtensorMap tmap_do,
                  const __grid_constant__ CUtensorMap tmap_o, int H, int N, int M, int G, int causal,
                  const __nv_bfloat16* __restrict__ q,
                  const __nv_bfloat16* __restrict__ k, const __nv_bfloat16* __restrict__ v,
                  const float* __restrict__ W1, const float* __restrict__ W2,
                  const __nv_bfloat16* __restrict__ outp, const float* __restrict__ den,
                  const __nv_bfloat16* __restrict__ dout, __nv_bfloat16* __restrict__ dq,
                  __nv_bfloat16* __restrict__ dk, __nv_bfloat16* __restrict__ dv,
                  float* __restrict__ dw_part,
                  const float* __restrict__ kw, const float* __restrict__ tau,
                  float* __restrict__ dtau_part, int units, int nsplit,
                  float* __restrict__ state_part, const float* __restrict__ state_total,
                  int* status)
{
    using L = BwCfg<NS>;
    // blocks [0, half): pass R, [half, 2 half): pass F, half = units * nsplit; within a pass
    // idx = (sequence * nsplit + split) * G + group (the groups of a cluster adjacent); the
    // chunks are split into nsplit ranges (non-causal modes; 1 for the causal scans).
    // Partial slots are indexed by slot = pass * half + idx.
    const int half_grid = units * nsplit;
    const int PASS = (int)blockIdx.x < half_grid ? kPassR : kPassF;
    const int idx = (int)blockIdx.x % half_grid;
    const int split = (idx / G) % nsplit;
    const int unit = (idx / G / nsplit) * G + idx % G;
    const int slot = PASS * half_grid + idx;
    __nv_bfloat16* const dx_out = PASS == kPassF ? dq : dk;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sb = smem_u32(sm);
    __shared__ uint32_t tmem_base_sh;
    __shared__ __align__(8) uint64_t mbar, tma_bar;
    // cluster exchange: xready: the partner's receive regions are free; xdone: the partner
    // has read what this CTA sent (so the staging region may be rewritten); xfull[0]: dq (F)
    // or dv (R) partial landed, xfull[1]: dk (R) (transaction counts)
    __shared__ __align__(8) uint64_t xready, xdone, xfull[2];
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wg = warp >> 2, quad = warp & 3, t = 32 * quad + lane;
    const int bh = unit / G, g = unit % G, h = bh % H;
    const size_t base = (size_t)bh * N * 64;
    float* zr = reinterpret_cast<float*>(sm + L::ZR);
    float* crow = reinterpret_cast<float*>(sm + L::CROW);
    float* spart = reinterpret_cast<float*>(sm + L::SPART);
    const float itau = KW ? expf(-tau[h]) : 0.f;
    // dtau = -sum_j ln(w_j) s_j with s_j = phi~(k_j) . dphi~(k_j) = dL / d ln(w_j).  Scaling
    // every key weight of a sequence by one factor leaves every output row unchanged, so the
    // s_j of a sequence sum to zero and any per-sequence constant may be subtracted from
    // ln(w_j); the log weight of the sequence's first key removes the common part, whose
    // terms would otherwise cancel only to the rounding of the s_j.
    const float lw0 = KW ? logf(kw[(size_t)bh * N]) : 0.f;
    float dtau_acc = 0.f;

    // ---- set-up: this group's projection rows, zero state, C16 ----
    for (int idx = tid; idx < L::P * 8; idx += kThreadsB) {
        const int r = idx >> 3, c = idx & 7, f = 64 * g + (r & 63);
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
        st_shared_v4(sb + L::W + swz128(r, c * 8), pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]),
                     pack_bf16(x[4], x[5]), pack_bf16(x[6], x[7]));
    }
    for (int idx = tid; idx < 16384 / 16; idx += kThreadsB) st_shared_v4(sb + L::SN + idx * 16, 0, 0, 0, 0);
    for (int idx = tid; idx < 4096 / 16; idx += kThreadsB) {
        const uint32_t fill = PASS == kPassF ? 0x3F803F80u : 0u;  // ones (z) or zeros (c rows)
        st_shared_v4(sb + L::C16 + idx * 16, fill, fill, fill, fill);
    }
    for (int idx = tid; idx < 128; idx += kThreadsB) zr[idx] = 0.f;
    const int rank = CS > 1 ? (int)cluster_rank() : 0;  // = g
    if (tid == 0) {
        mbar_init(&mbar, 1);
        mbar_init(&tma_bar, 1);
        mbar_init(&xready, 1);
        mbar_init(&xdone, 1);
        mbar_init(&xfull[0], 1);
        mbar_init(&xfull[1], 1);
        abort_flag = 0;
        fence_mbar_init();
        if (CS > 1) {  // the first chunk's exchanges
            mbar_arrive_expect_tx(&xfull[0], kXBytes);
            if (PASS == kPassR) mbar_arrive_expect_tx(&xfull[1], kXBytes);
        }
    }
    if (warp == 0) {
        tmem_alloc(&tmem_base_sh, 512);
        tmem_relinquish();
    }
    fence_proxy_async();
    fence_before_sync();
    if (CS > 1)
        cluster_sync();  // the partner's barriers exist before anything arrives on them
    else
        __syncthreads();
    fence_after_sync();
    const uint32_t tm = tmem_base_sh;
    const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);
    uint32_t phase = 0, tma_phase = 0, ph_xready = 0, ph_xdone = 0, ph_xfull[2] = {0, 0};
    const uint32_t partner = (uint32_t)rank ^ 1u;

    auto handoff = [&]() {
        fence_proxy_async();
        fence_before_sync();
        __syncthreads();
    };
    auto commit_wait = [&]() -> bool {  // thread 0 has issued MMAs: commit, all wait
        if (tid == 0) mma_commit(&mbar);
        bool ok = bar_wait(&mbar, phase, &abort_flag, status);
        phase ^= 1;
        ok = !__syncthreads_or(!ok);
        fence_after_sync();
        return ok;
    };
    auto adv = [](uint64_t d, uint32_t bytes) { return d + (bytes >> 4); };
    const uint64_t dQ = sdesc(sb + L::Q, 16, 1024), dK = sdesc(sb + L::K, 16, 1024);
    const uint64_t dV = sdesc(sb + L::V, 16, 1024), dG = sdesc(sb + L::GT, 16, 1024);
    const uint64_t dW = sdesc(sb + L::W, 16, 1024), dWmn = sdesc(sb + L::W, 16384, 1024);
    const uint64_t dPQ = sdesc(sb + L::PQ, 16, 1024), dPK = sdesc(sb + L::PK, 16, 1024);
    const uint64_t dPQmn = sdesc(sb + L::PQ, 16384, 1024), dPKmn = sdesc(sb + L::PK, 16384, 1024);
    const uint64_t dVmn = sdesc(sb + L::V, 16384, 1024), dGmn = sdesc(sb + L::GT, 16384, 1024);
    const uint64_t dQmn = sdesc(sb + L::Q, 16384, 1024), dKmn = sdesc(sb + L::K, 16384, 1024);
    const uint64_t dSN = sdesc(sb + L::SN, 16, 1024), dSNmn = sdesc(sb + L::SN, 16384, 1024);
    const uint64_t dC16 = sdesc(sb + L::C16, 16, 1024);
    const uint64_t dDAmn = sdesc(sb + L::Q, L::DA2 - L::Q, 1024);  // bf16(dA) as [query][key]
    const uint64_t dAmn = sdesc(sb + L::DO, L::O - L::DO, 1024);   // bf16(A)  as [query][key]
    constexpr uint32_t I_PROJ = idesc_bf16(128, L::P, 0, 0);
    constexpr uint32_t I_KK128 = idesc_bf16(128, 128, 0, 0);   // K-major A, K-major B, N=128
    constexpr uint32_t I_KM128 = idesc_bf16(128, 128, 0, 1);   // K-major A, MN-major B, N=128
    constexpr uint32_t I_MM128 = idesc_bf16(128, 128, 1, 1);   // MN-major A and B, N=128
    constexpr uint32_t I_KM64 = idesc_bf16(128, 64, 0, 1);
    constexpr uint32_t I_MM64 = idesc_bf16(128, 64, 1, 1);
    constexpr uint32_t I_M16 = idesc_bf16(128, 16, 1, 0);      // MN-major A, K-major B, N=16

    // projection of a tile into T_P, then features of this group into dst (K-major rows)
    auto issue_projection = [&](uint64_t dx, uint32_t col) {
#pragma unroll
        for (int ks = 0; ks < 4; ++ks)
            mma_bf16(tm + col, adv(dx, ks * 32), adv(dW, ks * 32), I_PROJ, ks > 0);
    };
    auto project = [&](uint64_t dx) {
        if (tid == 0) {
            fence_after_sync();
            issue_projection(dx, L::T_P);
        }
        return commit_wait();
    };
    // q into T_P and k into T_A (free until the attention MMAs), one round trip
    auto project_qk = [&]() {
        if (tid == 0) {
            fence_after_sync();
            issue_projection(dQ, L::T_P);
            issue_projection(dK, L::T_A);
        }
        return commit_wait();
    };
    auto features = [&](uint32_t dst, uint32_t tcol, bool valid, float wsc) {
        float a[32], w[32], m0, m1, m2 = 0.f, m3 = 0.f;  // m: max |x| per load
        tmem_ld16_maxabs(tm_row + tcol + 32 * wg, *reinterpret_cast<float(*)[16]>(&a[0]), m0);
        tmem_ld16_maxabs(tm_row + tcol + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&a[16]), m1);
        if (NS) {
            tmem_ld16_maxabs(tm_row + tcol + 64 + 32 * wg, *reinterpret_cast<float(*)[16]>(&w[0]), m2);
            tmem_ld16_maxabs(tm_row + tcol + 64 + 32 * wg + 16,
                             *reinterpret_cast<float(*)[16]>(&w[16]), m3);
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
            if (NS) {
                const float cw0 = w[2 * i], cw1 = w[2 * i + 1];
                c0 *= cw0; s0 *= cw0; c1 *= cw1; s1 *= cw1;
            }
            if (KW) { c0 *= wsc; s0 *= wsc; c1 *= wsc; s1 *= wsc; }
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
    };
    // Chain rule through the features of this thread's 32 frequencies: dphi from T_D plus
    // the per-feature term zr * scale, then da written over the feature tile in place
    // (s: da in the cos columns, zeros in the sin columns; n: du | dw).
    // wkey: the key weight (pass R with the prefactor, else 1); returns this thread's part
    // of s_t = phi~(k_t) . dphi~(k_t) (pass R with the prefactor, else 0).
    auto feature_backward = [&](uint32_t tile, float scale, bool valid, float wkey) -> float {
        float dc[32], ds[32];
        tmem_ld16(tm_row + L::T_D + 32 * wg, *reinterpret_cast<float(*)[16]>(&dc[0]));
        tmem_ld16(tm_row + L::T_D + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&dc[16]));
        tmem_ld16(tm_row + L::T_D + 64 + 32 * wg, *reinterpret_cast<float(*)[16]>(&ds[0]));
        tmem_ld16(tm_row + L::T_D + 64 + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&ds[16]));
        float a[32], w[32], m0 = 0.f, m1 = 0.f, m2 = 0.f, m3 = 0.f;  // m: max |x| per load
        if (NS) {  // u, w recomputed by a fresh projection in T_P
            tmem_ld16_maxabs(tm_row + L::T_P + 32 * wg, *reinterpret_cast<float(*)[16]>(&a[0]), m0);
            tmem_ld16_maxabs(tm_row + L::T_P + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&a[16]),
                             m1);
            tmem_ld16_maxabs(tm_row + L::T_P + 64 + 32 * wg, *reinterpret_cast<float(*)[16]>(&w[0]),
                             m2);
            tmem_ld16_maxabs(tm_row + L::T_P + 64 + 32 * wg + 16,
                             *reinterpret_cast<float(*)[16]>(&w[16]), m3);
        }
        tmem_wait_ld();
        if (NS) reduce_2pi_if_needed(a, w, fmaxf(fmaxf(m0, m1), fmaxf(m2, m3)));
        uint32_t cpair[16], spair[16];  // s: this thread's cos / sin features, bf16 pairs
        if (!NS) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const uint4 c4 = *reinterpret_cast<const uint4*>(sm + (tile - sb) + swz128(t, (4 * wg + j) * 8));
                const uint4 s4 =
                    *reinterpret_cast<const uint4*>(sm + (tile - sb) + 16384 + swz128(t, (4 * wg + j) * 8));
                cpair[4 * j] = c4.x; cpair[4 * j + 1] = c4.y; cpair[4 * j + 2] = c4.z; cpair[4 * j + 3] = c4.w;
                spair[4 * j] = s4.x; spair[4 * j + 1] = s4.y; spair[4 * j + 2] = s4.z; spair[4 * j + 3] = s4.w;
            }
        }
        float zc[32], zs[32];  // the per-feature term, z (pass F) or r (pass R)
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const float4 a4 = reinterpret_cast<const float4*>(zr + 32 * wg)[j];
            const float4 b4 = reinterpret_cast<const float4*>(zr + 64 + 32 * wg)[j];
            zc[4 * j] = a4.x; zc[4 * j + 1] = a4.y; zc[4 * j + 2] = a4.z; zc[4 * j + 3] = a4.w;
            zs[4 * j] = b4.x; zs[4 * j + 1] = b4.y; zs[4 * j + 2] = b4.z; zs[4 * j + 3] = b4.w;
        }
        const bool wt = KW && PASS == kPassR;
        float sdot = 0.f;
        uint32_t o1[16], o2[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            float r1[2], r2[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int fi = 2 * i + e;
                const float dphic = dc[fi] + scale * zc[fi], dphis = ds[fi] + scale * zs[fi];
                if (!NS) {  // the tile's features carry the key weight (pass R, prefactor)
                    const float pc = __uint_as_float(e ? cpair[i] & 0xFFFF0000u : cpair[i] << 16);
                    const float psn = __uint_as_float(e ? spair[i] & 0xFFFF0000u : spair[i] << 16);
                    r1[e] = -psn * dphic + pc * dphis;
                    r2[e] = 0.f;  // (the low bf16 part of da, set below)
                    if (wt) sdot = fmaf(pc, dphic, fmaf(psn, dphis, sdot));
                } else {
                    float su, cu, sw, cw;
                    __sincosf(a[fi], &su, &cu);
                    __sincosf(w[fi], &sw, &cw);
                    r1[e] = cw * (-su * dphic + cu * dphis);
                    r2[e] = -sw * (cu * dphic + su * dphis);
                    if (wt) {
                        sdot = fmaf(cu * cw, dphic, fmaf(su * cw, dphis, sdot));
                        r1[e] *= wkey;
                        r2[e] *= wkey;
                    }
                }
                if (!valid) r1[e] = r2[e] = 0.f;
            }
            o1[i] = pack_bf16(r1[0], r1[1]);
            if (!NS) {
                // s: the sin half of the tile (unused by dx = da W) carries da - bf16(da), so
                // the dW MMA (all 128 rows) gets da to ~2^-17: rows 64-127 of dW are added
                // to rows 0-63 in the reduction
                r2[0] = r1[0] - __uint_as_float(o1[i] << 16);
                r2[1] = r1[1] - __uint_as_float(o1[i] & 0xFFFF0000u);
            }
            o2[i] = pack_bf16(r2[0], r2[1]);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t off = swz128(t, (4 * wg + j) * 8);
            st_shared_v4(tile + off, o1[4 * j], o1[4 * j + 1], o1[4 * j + 2], o1[4 * j + 3]);
            st_shared_v4(tile + 16384 + off, o2[4 * j], o2[4 * j + 1], o2[4 * j + 2], o2[4 * j + 3]);
        }
        if (!valid) sdot = 0.f;
        return NS ? sdot * wkey : sdot;  // n: phi~ = w cos u cos w, w sin u cos w
    };
    // dx = da W (T_A[0,64)) and dW = da^T x: n: this chunk's in T_A[64,128); s: summed
    // over the chunks in the projection's unused half, T_P[64,128); n in kGrad: summed in
    // T_S, which holds no state without a scan
    constexpr bool kDwPerChunk = NS && MODE != kGrad;
    constexpr uint32_t T_DW = kDwPerChunk ? L::T_A + 64 : (NS ? L::T_S : L::T_P + 64);
    auto project_back = [&](uint64_t d_da, uint64_t d_da_mn, uint64_t d_x_mn, bool first) {
        if (tid == 0) {
            fence_after_sync();
            const int kst = NS ? 8 : 4;  // K = P rows of W (s: the cos half only)
            for (int ks = 0; ks < kst; ++ks)
                mma_bf16(tm + L::T_A, adv(d_da, (ks >> 2) * 16384 + (ks & 3) * 32),
                         adv(dWmn, ks * 2048), I_KM64, ks > 0);
#pragma unroll
            for (int ks = 0; ks < 8; ++ks)
                mma_bf16(tm + T_DW, adv(d_da_mn, ks * 2048), adv(d_x_mn, ks * 2048), I_MM64,
                         (kDwPerChunk ? ks > 0 : (!first || ks > 0)) ? 1u : 0u);
        }
        return commit_wait();
    };
    // dW rows of this chunk (lane = row of this group's projection) into the partial slot
    auto dw_accumulate = [&](bool first) {
        float v_[64];
#pragma unroll
        for (int j = 0; j < 4; ++j)
            tmem_ld16(tm_row + T_DW + 16 * j, *reinterpret_cast<float(*)[16]>(&v_[16 * j]));
        tmem_wait_ld();
        if (wg == 1) {  // all 128 rows (s: rows 64-127 hold the low part's contribution)
            float4* dst = reinterpret_cast<float4*>(dw_part + ((size_t)slot * 128 + t) * 64);
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                float4 old = first ? make_float4(0.f, 0.f, 0.f, 0.f) : dst[j];
                dst[j] = make_float4(old.x + v_[4 * j], old.y + v_[4 * j + 1],
                                     old.z + v_[4 * j + 2], old.w + v_[4 * j + 3]);
            }
        }
    };
    // state snapshot [feature][64] bf16 + column 64 (z or r) fp32, from T_S (lane = feature)
    auto snapshot = [&]() {
        float s_[32], zz[16];
        tmem_ld16(tm_row + L::T_S + 32 * wg, *reinterpret_cast<float(*)[16]>(&s_[0]));
        tmem_ld16(tm_row + L::T_S + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&s_[16]));
        tmem_ld16(tm_row + L::T_S + 64, zz);
        tmem_wait_ld();
#pragma unroll
        for (int j = 0; j < 4; ++j)
            st_shared_v4(sb + L::SN + swz128(t, (4 * wg + j) * 8),
                         pack_bf16(s_[8 * j], s_[8 * j + 1]), pack_bf16(s_[8 * j + 2], s_[8 * j + 3]),
                         pack_bf16(s_[8 * j + 4], s_[8 * j + 5]), pack_bf16(s_[8 * j + 6], s_[8 * j + 7]));
        if (wg == 0) zr[t] = zz[0];
    };
    // ---- cluster exchange of the dq / dk / dv partials (CS = 2) ----
    // This CTA's receive regions for the chunk are free: tell the partner (all threads are
    // past their last use of them).
    auto signal_ready = [&]() {
        if (CS > 1 && tid == 0) mbar_arrive_cluster(mapa(smem_u32(&xready), partner));
    };
    // Before the staging region is rewritten: the partner has read the previous chunk's data.
    auto wait_done = [&](bool any_sent) -> bool {
        bool ok = true;
        if (CS > 1 && any_sent && tid == 0) {
            ok = bar_wait_cluster(&xdone, ph_xdone, &abort_flag, status);
            ph_xdone ^= 1;
        }
        ok = !__syncthreads_or(!ok);
        return ok;
    };
    // Byte offset of 16-byte chunk j (0-7) of this thread's half row in a 64 x 64 fp32
    // exchange block (256-byte rows, chunks swizzled by row: conflict-free float4 access).
    auto xoff = [&](uint32_t rr, int j) {
        return rr * 256u + ((((uint32_t)(8 * wg + j)) ^ (rr & 7u)) << 4);
    };
    // Rows of a [128 x 64] TMEM block (T_A[0,64)) -> bf16 rows of `out` for the chunk at t0,
    // in two steps so that the exchange's latency is hidden behind other work.
    // send_rows: kcoef != 0 adds kcoef * k_t (the prefactor's dk term; k row from the K
    // tile).  Without a partner every row is stored at once.  With one, the rows the partner
    // finishes are staged at `stage` and bulk-copied to its `recv` (once it has signalled
    // that the region is free); this CTA's own rows (64 rank .. + 63) stay in T_A (written
    // back when the dk term was added) for finalize_rows.
    auto send_rows = [&](__nv_bfloat16* out, int t0, bool valid, float kcoef, int xi,
                         uint32_t stage, uint32_t recv) -> bool {
        float v_[32];
        tmem_ld16(tm_row + L::T_A + 32 * wg, *reinterpret_cast<float(*)[16]>(&v_[0]));
        tmem_ld16(tm_row + L::T_A + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&v_[16]));
        tmem_wait_ld();
        if (KW && kcoef != 0.f) {
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const uint4 k4 = *reinterpret_cast<const uint4*>(sm + L::K + swz128(t, 32 * wg + 8 * j));
                const uint32_t kw4[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    v_[8 * j + 2 * e] = fmaf(kcoef, __uint_as_float(kw4[e] << 16), v_[8 * j + 2 * e]);
                    v_[8 * j + 2 * e + 1] =
                        fmaf(kcoef, __uint_as_float(kw4[e] & 0xFFFF0000u), v_[8 * j + 2 * e + 1]);
                }
            }
        }
        bool ok = true;
        const bool own = CS == 1 || (t >> 6) == rank;  // uniform over a warp
        if (CS == 1) {
            if (valid) {
                uint4* dst = reinterpret_cast<uint4*>(out + base + (size_t)(t0 + t) * 64 + 32 * wg);
#pragma unroll
                for (int cc = 0; cc < 4; ++cc)
                    dst[cc] = make_uint4(pack_bf16(v_[8 * cc], v_[8 * cc + 1]),
                                         pack_bf16(v_[8 * cc + 2], v_[8 * cc + 3]),
                                         pack_bf16(v_[8 * cc + 4], v_[8 * cc + 5]),
                                         pack_bf16(v_[8 * cc + 6], v_[8 * cc + 7]));
            }
        } else {
            const uint32_t rr = (uint32_t)t & 63u;
            if (!own) {
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    st_shared_v4(stage + xoff(rr, j), __float_as_uint(v_[4 * j]),
                                 __float_as_uint(v_[4 * j + 1]), __float_as_uint(v_[4 * j + 2]),
                                 __float_as_uint(v_[4 * j + 3]));
            } else if (KW && xi == 1) {  // own dk rows keep the dk term
                uint32_t w_[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) w_[i] = __float_as_uint(v_[i]);
                tmem_st16(tm_row + L::T_A + 32 * wg, w_);
#pragma unroll
                for (int i = 0; i < 16; ++i) w_[i] = __float_as_uint(v_[16 + i]);
                tmem_st16(tm_row + L::T_A + 32 * wg + 16, w_);
                tmem_wait_st();
            }
            fence_proxy_async();  // the staged rows, visible to the bulk copy
            fence_before_sync();
            __syncthreads();
            if (tid == 0) {
                if (xi == 0) {  // one "ready" per chunk covers its exchanges
                    ok = bar_wait_cluster(&xready, ph_xready, &abort_flag, status);
                    ph_xready ^= 1;
                }
                if (ok)
                    bulk_copy_cluster(mapa(recv, partner), stage, kXBytes,
                                      mapa(smem_u32(&xfull[xi]), partner));
            }
        }
        fence_proxy_async();  // generic reads of the K tile before its next TMA load
        ok = !__syncthreads_or(!ok);
        fence_after_sync();
        return ok;
    };
    // finalize_rows (with a partner): once the partner's partial of this CTA's own rows has
    // landed at `recv`, adds it to the rows still in T_A and stores bf16 rows of the chunk at
    // t0 (CL valid rows); re-arms exchange xi for the next chunk and, after the chunk's last
    // exchange, tells the partner that its staging region may be rewritten.
    auto finalize_rows = [&](__nv_bfloat16* out, int t0, int CL, int xi, uint32_t recv,
                             bool last) -> bool {
        if (CS == 1) return true;
        bool ok = true;
        if ((t >> 6) == rank) {  // uniform over a warp
            const uint32_t rr = (uint32_t)t & 63u;
            float v_[32];
            tmem_ld16(tm_row + L::T_A + 32 * wg, *reinterpret_cast<float(*)[16]>(&v_[0]));
            tmem_ld16(tm_row + L::T_A + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&v_[16]));
            ok = bar_wait(&xfull[xi], ph_xfull[xi], &abort_flag, status);
            tmem_wait_ld();
            if (ok) {
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const float4 p4 = *reinterpret_cast<const float4*>(sm + (recv - sb) + xoff(rr, j));
                    v_[4 * j] += p4.x;
                    v_[4 * j + 1] += p4.y;
                    v_[4 * j + 2] += p4.z;
                    v_[4 * j + 3] += p4.w;
                }
                if (t < CL) {
                    uint4* dst = reinterpret_cast<uint4*>(out + base + (size_t)(t0 + t) * 64 + 32 * wg);
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc)
                        dst[cc] = make_uint4(pack_bf16(v_[8 * cc], v_[8 * cc + 1]),
                                             pack_bf16(v_[8 * cc + 2], v_[8 * cc + 3]),
                                             pack_bf16(v_[8 * cc + 4], v_[8 * cc + 5]),
                                             pack_bf16(v_[8 * cc + 6], v_[8 * cc + 7]));
                }
            }
        }
        ph_xfull[xi] ^= 1;
        fence_before_sync();
        ok = !__syncthreads_or(!ok);
        fence_after_sync();
        if (ok && tid == 0) {
            mbar_arrive_expect_tx(&xfull[xi], kXBytes);
            if (last) mbar_arrive_cluster(mapa(smem_u32(&xdone), partner));
        }
        return ok;
    };
    const float dscale = 1.0f / (float)M;  // den' = M den
    // g = dout / den' (bf16, the tile GT) and c_t = -(g . out) (crow; with c_row also row 0
    // of the c operand C16, and with c_lo row 1 = c - bf16(c)) from the dout and out tiles;
    // each thread takes half a row.
    auto build_g = [&](bool valid_, float den_t, bool c_row, bool c_lo) {
        {
            const float gsc = valid_ ? dscale / den_t : 0.f;
            float dot = 0.f;
            uint32_t gp[16];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int cc = 4 * wg + j;
                const uint4 a4 = *reinterpret_cast<const uint4*>(sm + L::DO + swz128(t, cc * 8));
                const uint4 o4 = *reinterpret_cast<const uint4*>(sm + L::O + swz128(t, cc * 8));
                const uint32_t aw[4] = {a4.x, a4.y, a4.z, a4.w}, ow[4] = {o4.x, o4.y, o4.z, o4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float a0 = __uint_as_float(aw[e] << 16), a1 = __uint_as_float(aw[e] & 0xFFFF0000u);
                    const float b0 = __uint_as_float(ow[e] << 16), b1 = __uint_as_float(ow[e] & 0xFFFF0000u);
                    // c uses the same bf16-rounded g as the MMAs, so g.v_j + c_i cancels
                    // exactly where out_i = v_j (e.g. the first causal position)
                    const uint32_t gw = pack_bf16(a0 * gsc, a1 * gsc);
                    gp[j * 4 + e] = gw;
                    dot = fmaf(__uint_as_float(gw << 16), b0,
                               fmaf(__uint_as_float(gw & 0xFFFF0000u), b1, dot));
                }
            }
#pragma unroll
            for (int j = 0; j < 4; ++j)
                st_shared_v4(sb + L::GT + swz128(t, (4 * wg + j) * 8), gp[4 * j], gp[4 * j + 1],
                             gp[4 * j + 2], gp[4 * j + 3]);
            spart[128 * wg + t] = dot;  // free until the feature backward
        }
        handoff();
        if (wg == 0) {
            const float cval = valid_ ? -(spart[t] + spart[128 + t]) : 0.f;
            crow[t] = cval;
            if (c_row) {  // row 0 of the K-major [16][tokens] c operand
                const __nv_bfloat16 chi = __float2bfloat16_rn(cval);
                *reinterpret_cast<__nv_bfloat16*>(sm + L::C16 + (t >> 6) * 2048 + swz128(0, t & 63)) = chi;
                if (c_lo)
                    *reinterpret_cast<__nv_bfloat16*>(sm + L::C16 + (t >> 6) * 2048 + swz128(1, t & 63)) =
                        __float2bfloat16_rn(cval - __bfloat162float(chi));
            }
        }
    };
    // TMA of one tile of chunk cn into shared memory (completes on tma_bar)
    auto load_tile = [&](uint32_t dst, const CUtensorMap* map, int cn) {
        tma_load_3d(sb + dst, map, 0, cn * kC, bh, &tma_bar);
    };

    const int nch = (N + kC - 1) / kC;
    int prev_t0 = 0, prev_CL = 0;  // the chunk whose dq (F) or dk (R) rows await the partner
    bool tma_outstanding = false;  // tile loads issued and not yet waited for
    if constexpr (MODE == kCausal) {
    // Tiles of chunk c + 1 are loaded while chunk c is worked on, each as soon as its region
    // is free: pass F: dout, out after g is built, k after the projections, v after the state
    // update, q after the projection backward; pass R: q, v, dout, out after the gradient
    // MMAs, k once the dk rows are sent.  All five complete on tma_bar.
    if (tid == 0) {
        const int c0 = PASS == kPassF ? 0 : nch - 1;
        mbar_arrive_expect_tx(&tma_bar, 5 * kTileBytes);
        load_tile(L::Q, &tmap_q, c0);
        load_tile(L::K, &tmap_k, c0);
        load_tile(L::V, &tmap_v, c0);
        load_tile(L::DO, &tmap_do, c0);
        load_tile(L::O, &tmap_o, c0);
    }
    tma_outstanding = true;
    for (int it = 0; it < nch; ++it) {
        const int c = PASS == kPassF ? it : nch - 1 - it;
        const int cn = PASS == kPassF ? c + 1 : c - 1;  // the next chunk, if it exists
        const bool has_next = it + 1 < nch;
        const int t0 = c * kC, CL = min(kC, N - t0);
        const bool valid = t < CL;
        const float wk = (KW && valid) ? kw[(size_t)bh * N + t0 + t] : 1.f;
        if (tid == 0 && it + 2 < nch) {  // the chunk after next into L2
            const int c2 = PASS == kPassF ? c + 2 : c - 2;
            const size_t off = base + (size_t)c2 * kC * 64;
            const uint32_t bytes = (uint32_t)min(kC, N - c2 * kC) * 128;
            prefetch_l2(q + off, bytes);
            prefetch_l2(k + off, bytes);
            prefetch_l2(v + off, bytes);
            prefetch_l2(dout + off, bytes);
            prefetch_l2(outp + off, bytes);
        }
        // ---- this chunk's tiles (rows past N read as zero); then the g tile and c_t from
        // dout, out (shared memory) and den, each thread taking half a row ----
        const float den_t = valid ? den[(size_t)bh * N + t0 + t] : 1.f;
        if (!bar_wait(&tma_bar, tma_phase, &abort_flag, status)) goto done;
        tma_phase ^= 1;
        tma_outstanding = false;
        // pass R: the previous chunk's dk rows (received in GT, which g overwrites next)
        if (PASS == kPassR && it > 0 &&
            !finalize_rows(dx_out, prev_t0, prev_CL, 1, sb + L::GT, true))
            goto done;
        build_g(valid, den_t, PASS == kPassR, false);
        if (PASS == kPassF) {
            if (tid == 0 && has_next) {  // DO, O are free: the next chunk's dout, out
                mbar_arrive_expect_tx(&tma_bar, 5 * kTileBytes);
                load_tile(L::DO, &tmap_do, cn);
                load_tile(L::O, &tmap_o, cn);
            }
            tma_outstanding = has_next;
            // the previous chunk's dq rows (received in PK, which the features overwrite)
            if (it > 0 && !finalize_rows(dx_out, prev_t0, prev_CL, 0, sb + L::PK, true)) goto done;
        }
        // ---- features of q and k for this group ----
        if (!project_qk()) goto done;
        if (PASS == kPassF && tid == 0 && has_next) load_tile(L::K, &tmap_k, cn);  // K is free
        // the partner has read the previous chunk's exchange data staged in PQ
        if (CS > 1 && !wait_done(it > 0)) goto done;
        features(sb + L::PQ, L::T_P, valid, 1.f);
        features(sb + L::PK, L::T_A, valid, wk);
        handoff();

        if (PASS == kPassF) {
            // dA = g v^T, then + c, mask, bf16 in place (A operand of dphi(q) = dA phi(K))
            if (tid == 0) {
                fence_after_sync();
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_bf16(tm + L::T_A, adv(dG, ks * 32), adv(dV, ks * 32), I_KK128, ks > 0);
            }
            if (!commit_wait()) goto done;
            {
                const float cv = crow[t];
#pragma unroll
                for (int b = 0; b < 2; ++b) {
                    const uint32_t col = L::T_A + 64 * wg + 32 * b;
                    float a[32];
                    tmem_ld16(tm_row + col, *reinterpret_cast<float(*)[16]>(&a[0]));
                    tmem_ld16(tm_row + col + 16, *reinterpret_cast<float(*)[16]>(&a[16]));
                    tmem_wait_ld();
                    uint32_t pk2[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int j0 = 64 * wg + 32 * b + 2 * i;
                        const bool m0 = (!causal || j0 <= t) && j0 < CL && valid;
                        const bool m1 = (!causal || j0 + 1 <= t) && j0 + 1 < CL && valid;
                        pk2[i] = pack_bf16(m0 ? a[2 * i] + cv : 0.f, m1 ? a[2 * i + 1] + cv : 0.f);
                    }
                    tmem_st16(tm_row + L::T_A + 64 * wg + 16 * b, pk2);
                }
                tmem_wait_st();
            }
            handoff();
            // dphi(q) = dA phi(K) + g S^T; S += phi(K)^T v; z += phi(K)^T 1
            if (tid == 0) {
                fence_after_sync();
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_bf16_tmem_a(tm + L::T_D, tm + L::T_A + 64 * (ks >> 2) + 8 * (ks & 3),
                                    adv(dPKmn, ks * 2048), I_KM128, ks > 0);
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_bf16(tm + L::T_D, adv(dG, ks * 32), adv(dSN, ks * 32), I_KK128, 1u);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {
                    const uint32_t acc = (it > 0 || ks > 0) ? 1u : 0u;
                    mma_bf16(tm + L::T_S, adv(dPKmn, ks * 2048), adv(dVmn, ks * 2048), I_MM64, acc);
                    mma_bf16(tm + L::T_S + 64, adv(dPKmn, ks * 2048),
                             adv(dC16, (ks >> 2) * 2048 + (ks & 3) * 32), I_M16, acc);
                }
            }
            if (!commit_wait()) goto done;
            signal_ready();  // PK is free for the partner's dq partial
            if (tid == 0 && has_next) load_tile(L::V, &tmap_v, cn);  // V is free
            // n: u, w of q for the chain rule are still in T_P
            feature_backward(sb + L::PQ, crow[t], valid, 1.f);
            handoff();
            if (!project_back(dPQ, dPQmn, dQmn, it == 0)) goto done;
            if (tid == 0 && has_next) load_tile(L::Q, &tmap_q, cn);  // Q is free
            if (!send_rows(dx_out, t0, valid, 0.f, 0, sb + L::PQ, sb + L::PK)) goto done;
            prev_t0 = t0;
            prev_CL = CL;
            if (NS) dw_accumulate(it == 0);
            snapshot();
            handoff();
        } else {
            // A = phi(Q) phi(K)^T -> mask -> bf16 [query][key] in [DO | O]
            if (tid == 0) {
                fence_after_sync();
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {
                    const uint32_t kofs = (ks >> 2) * 16384 + (ks & 3) * 32;
                    mma_bf16(tm + L::T_A, adv(dPQ, kofs), adv(dPK, kofs), I_KK128, ks > 0);
                }
            }
            if (!commit_wait()) goto done;
            auto mask_to_smem = [&](uint32_t blk0, float add) {
#pragma unroll
                for (int b = 0; b < 2; ++b) {
                    float a[32];
                    tmem_ld16(tm_row + L::T_A + 64 * wg + 32 * b, *reinterpret_cast<float(*)[16]>(&a[0]));
                    tmem_ld16(tm_row + L::T_A + 64 * wg + 32 * b + 16,
                              *reinterpret_cast<float(*)[16]>(&a[16]));
                    tmem_wait_ld();
                    uint32_t pk2[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int j0 = 64 * wg + 32 * b + 2 * i;
                        const bool m0 = (!causal || j0 <= t) && j0 < CL && valid;
                        const bool m1 = (!causal || j0 + 1 <= t) && j0 + 1 < CL && valid;
                        pk2[i] = pack_bf16(m0 ? a[2 * i] + add : 0.f, m1 ? a[2 * i + 1] + add : 0.f);
                    }
                    const uint32_t dst = blk0 + wg * 16384;  // key block wg
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        st_shared_v4(dst + swz128(t, (4 * b + j) * 8), pk2[4 * j], pk2[4 * j + 1],
                                     pk2[4 * j + 2], pk2[4 * j + 3]);
                }
            };
            mask_to_smem(sb + L::DO, 0.f);
            fence_before_sync();
            __syncthreads();
            // dA = g v^T -> + c, mask -> bf16 [query][key] in [Q | DA2]
            if (tid == 0) {
                fence_after_sync();
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_bf16(tm + L::T_A, adv(dG, ks * 32), adv(dV, ks * 32), I_KK128, ks > 0);
            }
            if (!commit_wait()) goto done;
            mask_to_smem(sb + L::Q, crow[t]);
            handoff();
            // dphi(k) = dA^T phi(Q) + v R^T;  dv = A^T g + phi(K) R;  R += phi(Q)^T g;
            // r += phi(Q)^T c
            if (tid == 0) {
                fence_after_sync();
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_bf16(tm + L::T_D, adv(dDAmn, ks * 2048), adv(dPQmn, ks * 2048), I_MM128, ks > 0);
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_bf16(tm + L::T_D, adv(dV, ks * 32), adv(dSN, ks * 32), I_KK128, 1u);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_bf16(tm + L::T_A, adv(dAmn, ks * 2048), adv(dGmn, ks * 2048), I_MM64, ks > 0);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks)
                    mma_bf16(tm + L::T_A, adv(dPK, (ks >> 2) * 16384 + (ks & 3) * 32),
                             adv(dSNmn, ks * 2048), I_KM64, 1u);
#pragma unroll
                for (int ks = 0; ks < 8; ++ks) {
                    const uint32_t acc = (it > 0 || ks > 0) ? 1u : 0u;
                    mma_bf16(tm + L::T_S, adv(dPQmn, ks * 2048), adv(dGmn, ks * 2048), I_MM64, acc);
                    mma_bf16(tm + L::T_S + 64, adv(dPQmn, ks * 2048),
                             adv(dC16, (ks >> 2) * 2048 + (ks & 3) * 32), I_M16, acc);
                }
            }
            if (!commit_wait()) goto done;
            signal_ready();  // DA2, GT are free for the partner's dv, dk partials
            if (tid == 0 && has_next) {  // Q, V, DO, O are free: the next chunk's tiles
                mbar_arrive_expect_tx(&tma_bar, 5 * kTileBytes);
                load_tile(L::Q, &tmap_q, cn);
                load_tile(L::V, &tmap_v, cn);
                load_tile(L::DO, &tmap_do, cn);
                load_tile(L::O, &tmap_o, cn);
            }
            tma_outstanding = has_next;
            // dv of this group: sent now, finished before the projection backward overwrites it
            if (!send_rows(dv, t0, valid, 0.f, 0, sb + L::PQ, sb + L::DA2)) goto done;
            if (NS && !project(dK)) goto done;  // u, w of k for the chain rule
            {
                const float sp = feature_backward(sb + L::PK, 1.0f, valid, wk);
                if (KW) {
                    spart[128 * wg + t] = sp;
                    // ln w = |k|^2 exp(-tau), centred on the sequence's first key (the s_j of
                    // a sequence sum to zero): the cancelling part drops out exactly
                    dtau_acc = fmaf(lw0 - logf(wk), sp, dtau_acc);
                }
            }
            handoff();
            if (!finalize_rows(dv, t0, CL, 0, sb + L::DA2, false)) goto done;
            if (!project_back(dPK, dPKmn, dKmn, it == 0)) goto done;
            if (!send_rows(dx_out, t0, valid, KW ? 2.f * itau * (spart[t] + spart[128 + t]) : 0.f,
                           1, sb + L::PQ + 16384, sb + L::GT))
                goto done;
            if (tid == 0 && has_next) load_tile(L::K, &tmap_k, cn);  // K is free
            prev_t0 = t0;
            prev_CL = CL;
            if (NS) dw_accumulate(it == 0);
            snapshot();
            handoff();
        }
    }
    // the last chunk's rows that await the partner: dq (F) or dk (R)
    if (!finalize_rows(dx_out, prev_t0, prev_CL, PASS == kPassF ? 0 : 1,
                       sb + (PASS == kPassF ? L::PK : L::GT), false))
        goto done;
    } else {
        // ---- non-causal: the chunks [cbeg, cend) of this split, in order ----
        const int cps = (nch + nsplit - 1) / nsplit;
        const int cbeg = split * cps, cend = min(nch, cbeg + cps);
        // this CTA reads q, dout, out (kState R, kGrad F) or k, v (kState F, kGrad R)
        const bool fq = (MODE == kState) == (PASS == kPassR);
        // kGrad: the low part of the state snapshot, in a region the pass does not use
        const uint32_t sl = sb + (PASS == kPassF ? L::V : L::PQ);
        const uint64_t dSL = sdesc(sl, 16, 1024), dSLmn = sdesc(sl, 16384, 1024);
        if (MODE == kGrad) {
            // the totals ([S | z] for pass F, [R | r] for pass R) as the state snapshot, split
            // into bf16 high (SN) and low (SL) parts [feature][64] so that the two MMAs carry
            // the fp32 totals to ~2^-17: the terms S g and c z (R v and r) cancel exactly
            // where the result is 0 (e.g. dq at N = 1); column 64 in zr (fp32)
            const float* st = state_total + ((size_t)PASS * units + unit) * 128 * 80 + (size_t)t * 80;
            float s_[32];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const float4 f4 = reinterpret_cast<const float4*>(st + 32 * wg)[j];
                s_[4 * j] = f4.x; s_[4 * j + 1] = f4.y; s_[4 * j + 2] = f4.z; s_[4 * j + 3] = f4.w;
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                uint32_t hi[4], lo[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float x0 = s_[8 * j + 2 * e], x1 = s_[8 * j + 2 * e + 1];
                    hi[e] = pack_bf16(x0, x1);
                    lo[e] = pack_bf16(x0 - __uint_as_float(hi[e] << 16),
                                      x1 - __uint_as_float(hi[e] & 0xFFFF0000u));
                }
                const uint32_t off = swz128(t, (4 * wg + j) * 8);
                st_shared_v4(sb + L::SN + off, hi[0], hi[1], hi[2], hi[3]);
                st_shared_v4(sl + off, lo[0], lo[1], lo[2], lo[3]);
            }
            if (wg == 0) zr[t] = st[64];
            signal_ready();  // this CTA's receive regions are free for the first exchange
        }
        // The tiles of chunk c + 1 are loaded while chunk c is worked on, each as soon as its
        // region is free: dout, out once g is built, q after its last MMA (the projection,
        // or in kGrad the projection backward); k after its projection (kState) or once the
        // dk rows are sent (kGrad), v after the MMA that reads it.
        const uint32_t nc_bytes = (fq ? 3 : 2) * kTileBytes;
        if (tid == 0 && cbeg < cend) {
            mbar_arrive_expect_tx(&tma_bar, nc_bytes);
            if (fq) {
                load_tile(L::Q, &tmap_q, cbeg);
                load_tile(L::DO, &tmap_do, cbeg);
                load_tile(L::O, &tmap_o, cbeg);
            } else {
                load_tile(L::K, &tmap_k, cbeg);
                load_tile(L::V, &tmap_v, cbeg);
            }
        }
        tma_outstanding = cbeg < cend;
        for (int c = cbeg; c < cend; ++c) {
            const int it = c - cbeg;
            const bool has_next = c + 1 < cend;
            const int t0 = c * kC, CL = min(kC, N - t0);
            const bool valid = t < CL;
            const float wk = (KW && !fq && valid) ? kw[(size_t)bh * N + t0 + t] : 1.f;
            const float den_t = (fq && valid) ? den[(size_t)bh * N + t0 + t] : 1.f;
            if (tid == 0 && c + 2 < cend) {  // the chunk after next into L2
                const size_t off = base + (size_t)(c + 2) * kC * 64;
                const uint32_t bytes = (uint32_t)min(kC, N - (c + 2) * kC) * 128;
                if (fq) {
                    prefetch_l2(q + off, bytes);
                    prefetch_l2(dout + off, bytes);
                    prefetch_l2(outp + off, bytes);
                } else {
                    prefetch_l2(k + off, bytes);
                    prefetch_l2(v + off, bytes);
                }
            }
            // arms the next chunk's loads at its first issue point
            auto arm_next = [&]() {
                if (tid == 0 && has_next) mbar_arrive_expect_tx(&tma_bar, nc_bytes);
                tma_outstanding = has_next;
            };
            if (!bar_wait(&tma_bar, tma_phase, &abort_flag, status)) goto done;
            tma_phase ^= 1;
            tma_outstanding = false;
            // g, c (and for the state [R | r] the c rows of C16: high and low bf16 parts, so r
            // carries c to ~2^-17 like the exact-cancelling term g . v)
            if (fq) {
                build_g(valid, den_t, PASS == kPassR, MODE == kState);
                arm_next();
                if (tid == 0 && has_next) {  // DO, O are free
                    load_tile(L::DO, &tmap_do, c + 1);
                    load_tile(L::O, &tmap_o, c + 1);
                }
            }
            // ---- features of the tile's rows (q or k) for this group ----
            if (!project(fq ? dQ : dK)) goto done;
            if (MODE == kState) {  // the projection was the tile's last use
                if (!fq) arm_next();
                if (tid == 0 && has_next) load_tile(fq ? L::Q : L::K, fq ? &tmap_q : &tmap_k, c + 1);
            }
            features(fq ? sb + L::PQ : sb + L::PK, L::T_P, valid, fq ? 1.f : wk);
            handoff();
            if (MODE == kState) {
                // [S | z] += phi(K)^T [V | 1]  or  [R | r] += phi(Q)^T [G | c]
                if (tid == 0) {
                    fence_after_sync();
                    const uint64_t dphi = fq ? dPQmn : dPKmn, dval = fq ? dGmn : dVmn;
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks) {
                        const uint32_t acc = (it > 0 || ks > 0) ? 1u : 0u;
                        mma_bf16(tm + L::T_S, adv(dphi, ks * 2048), adv(dval, ks * 2048), I_MM64, acc);
                        mma_bf16(tm + L::T_S + 64, adv(dphi, ks * 2048),
                                 adv(dC16, (ks >> 2) * 2048 + (ks & 3) * 32), I_M16, acc);
                    }
                }
                if (!commit_wait()) goto done;
                if (!fq && tid == 0 && has_next) load_tile(L::V, &tmap_v, c + 1);  // V is free
                continue;
            }
            if (PASS == kPassF) {
                // dphi(q) = g S^T (+ c z in the feature backward)
                if (tid == 0) {
                    fence_after_sync();
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        mma_bf16(tm + L::T_D, adv(dG, ks * 32), adv(dSN, ks * 32), I_KK128, ks > 0);
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        mma_bf16(tm + L::T_D, adv(dG, ks * 32), adv(dSL, ks * 32), I_KK128, 1u);
                }
                if (!commit_wait()) goto done;
                // n: u, w of q for the chain rule are still in T_P
                feature_backward(sb + L::PQ, crow[t], valid, 1.f);
                handoff();
                // the previous chunk's dq rows (received in PK), before the projection
                // backward overwrites them; PK is then free for this chunk's exchange
                if (it > 0) {
                    if (!finalize_rows(dx_out, prev_t0, prev_CL, 0, sb + L::PK, true)) goto done;
                    signal_ready();
                }
                if (!project_back(dPQ, dPQmn, dQmn, it == 0)) goto done;
                if (tid == 0 && has_next) load_tile(L::Q, &tmap_q, c + 1);  // Q is free
                // the partner has read the previous chunk's rows staged in K
                if (CS > 1 && !wait_done(it > 0)) goto done;
                if (!send_rows(dx_out, t0, valid, 0.f, 0, sb + L::K, sb + L::PK)) goto done;
                prev_t0 = t0;
                prev_CL = CL;
                if (kDwPerChunk) dw_accumulate(it == 0);
                handoff();
            } else {
                // the previous chunk's dk rows (received in O), before T_A is overwritten;
                // DO, O are then free for this chunk's exchanges
                if (it > 0) {
                    if (!finalize_rows(dx_out, prev_t0, prev_CL, 1, sb + L::O, true)) goto done;
                    signal_ready();
                }
                // dphi(k) = v R^T (+ r in the feature backward);  dv = phi(K) R
                if (tid == 0) {
                    fence_after_sync();
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        mma_bf16(tm + L::T_D, adv(dV, ks * 32), adv(dSN, ks * 32), I_KK128, ks > 0);
#pragma unroll
                    for (int ks = 0; ks < 4; ++ks)
                        mma_bf16(tm + L::T_D, adv(dV, ks * 32), adv(dSL, ks * 32), I_KK128, 1u);
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        mma_bf16(tm + L::T_A, adv(dPK, (ks >> 2) * 16384 + (ks & 3) * 32),
                                 adv(dSNmn, ks * 2048), I_KM64, ks > 0);
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)
                        mma_bf16(tm + L::T_A, adv(dPK, (ks >> 2) * 16384 + (ks & 3) * 32),
                                 adv(dSLmn, ks * 2048), I_KM64, 1u);
                }
                if (!commit_wait()) goto done;
                arm_next();
                if (tid == 0 && has_next) load_tile(L::V, &tmap_v, c + 1);  // V is free
                // the partner has read the previous chunk's rows staged in Q and DA2
                if (CS > 1 && !wait_done(it > 0)) goto done;
                if (!send_rows(dv, t0, valid, 0.f, 0, sb + L::Q, sb + L::DO)) goto done;
                {  // n: u, w of k for the chain rule are still in T_P
                    const float sp = feature_backward(sb + L::PK, 1.0f, valid, wk);
                    if (KW) {
                        spart[128 * wg + t] = sp;
                        // ln w = |k|^2 exp(-tau), centred on the sequence's first key (the s_j of
                    // a sequence sum to zero): the cancelling part drops out exactly
                    dtau_acc = fmaf(lw0 - logf(wk), sp, dtau_acc);
                    }
                }
                handoff();
                if (!finalize_rows(dv, t0, CL, 0, sb + L::DO, false)) goto done;
                if (!project_back(dPK, dPKmn, dKmn, it == 0)) goto done;
                if (!send_rows(dx_out, t0, valid, KW ? 2.f * itau * (spart[t] + spart[128 + t]) : 0.f,
                               1, sb + L::DA2, sb + L::O))
                    goto done;
                if (tid == 0 && has_next) load_tile(L::K, &tmap_k, c + 1);  // K is free
                prev_t0 = t0;
                prev_CL = CL;
                if (kDwPerChunk) dw_accumulate(it == 0);
                handoff();
            }
        }
        if (MODE == kState) {
            // this CTA's partial state [128 features][80] fp32: S (or R) in columns 0-63,
            // z (or r) in column 64
            float s_[32], zz[16];
            tmem_ld16(tm_row + L::T_S + 32 * wg, *reinterpret_cast<float(*)[16]>(&s_[0]));
            tmem_ld16(tm_row + L::T_S + 32 * wg + 16, *reinterpret_cast<float(*)[16]>(&s_[16]));
            tmem_ld16(tm_row + L::T_S + 64, zz);
            tmem_wait_ld();
            float* dst = state_part + ((size_t)slot * 128 + t) * 80;
#pragma unroll
            for (int j = 0; j < 8; ++j)
                reinterpret_cast<float4*>(dst + 32 * wg)[j] =
                    make_float4(s_[4 * j], s_[4 * j + 1], s_[4 * j + 2], s_[4 * j + 3]);
            // r = column 64 (c high) + column 65 (c low); z: column 64 (every C16 row is 1)
            if (wg == 0) dst[64] = PASS == kPassR ? zz[0] + zz[1] : zz[0];
        } else if (!finalize_rows(dx_out, prev_t0, prev_CL, PASS == kPassF ? 0 : 1,
                                  sb + (PASS == kPassF ? L::PK : L::O), false)) {
            goto done;  // the last chunk's dq (F) or dk (R) rows
        }
    }
    // s (and n in kGrad): the sum over the chunks, held in tensor memory
    if (MODE != kState && !kDwPerChunk) dw_accumulate(true);
    if (KW && MODE != kState) {  // this CTA's dtau (pass R; 0 in pass F): warps, then in order
        for (int o = 16; o > 0; o >>= 1) dtau_acc += __shfl_xor_sync(0xffffffffu, dtau_acc, o);
        __syncthreads();
        if (lane == 0) spart[warp] = dtau_acc;
        __syncthreads();
        if (tid == 0) {
            float sum = 0.f;
            for (int w8 = 0; w8 < kThreadsB / 32; ++w8) sum += spart[w8];
            dtau_part[slot] = sum;
        }
    }
done:
    if (abort_flag && tid == 0) {  // gave up: let copies into this CTA's shared memory land
        if (tma_outstanding) mbar_drain(&tma_bar, tma_phase, kDrainCycles);
        if (CS > 1) {
            mbar_drain(&xfull[0], ph_xfull[0], kDrainCycles);
            if (PASS == kPassR) mbar_drain(&xfull[1], ph_xfull[1], kDrainCycles);
        }
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == 0) tmem_dealloc(tm, 512);
    if (CS > 1) cluster_sync();  // no CTA leaves while its partner may still copy into it
}

// dW over the batch (and the chunk splits) in a fixed order.  Partial slots
// [pass][((b * H + h) * nsplit + s) * G + g][row][64]; s: rows < 64 are frequencies
// 64g + row (from the high bf16 part of da), rows >= 64 the same frequencies (from its low
// part); n: rows < 64 are dU, rows >= 64 are dV of frequency 64g + row%64.
__global__ void tc_dw_reduce_kernel(int B, int H, int M, int G, int nsplit, int nonstat,
                                    const float* __restrict__ part, float* __restrict__ dW1,
                                    float* __restrict__ dW2, const float* __restrict__ dtau_part,
                                    float* __restrict__ dtau)
{
    const size_t half = (size_t)B * H * nsplit * G;  // slots per pass
    if (dtau && blockIdx.x == 0)  // dtau[h]: the pass R slots of head h, in order
        for (int h = threadIdx.x; h < H; h += blockDim.x) {
            float a = 0.f;
            for (int b = 0; b < B; ++b)
                for (int sp = 0; sp < nsplit; ++sp)
                    for (int g = 0; g < G; ++g)
                        a += dtau_part[half + ((size_t)(b * H + h) * nsplit + sp) * G + g];
            dtau[h] = a;
        }
    const size_t total = (size_t)H * M * 64;
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int h = (int)(idx / ((size_t)M * 64));
        const int f = (int)((idx / 64) % M), e = (int)(idx % 64);
        const int g = f / 64, r = f % 64;
        float a = 0.f, b2 = 0.f;
        const size_t pass_stride = half * 128 * 64;  // pass F slots follow pass R's
        for (int b = 0; b < B; ++b)
            for (int sp = 0; sp < nsplit; ++sp) {
                const float* p = part + ((((size_t)(b * H + h) * nsplit + sp) * G + g) * 128) * 64;
                a += p[(size_t)r * 64 + e] + p[pass_stride + (size_t)r * 64 + e];
                // n: dV rows; s: the dW rows of the low part of da
                b2 += p[(size_t)(64 + r) * 64 + e] + p[pass_stride + (size_t)(64 + r) * 64 + e];
            }
        if (!nonstat) {
            dW1[idx] = a + b2;
        } else {
            dW1[idx] = 0.5f * (a + b2);
            dW2[idx] = 0.5f * (a - b2);
        }
    }
}

// Non-causal totals: total[pass][unit][row][0..64] = sum over the splits, in order, of the
// partial states [pass][(bh * nsplit + s) * G + g][row][0..64] (unit = bh * G + g).
__global__ void nc_state_reduce_kernel(int units, int G, int nsplit,
                                       const float* __restrict__ part, float* __restrict__ total)
{
    const size_t n = (size_t)2 * units * 128 * 65;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (size_t)gridDim.x * blockDim.x) {
        const int col = (int)(i % 65), row = (int)((i / 65) % 128);
        const int u = (int)((i / (65 * 128)) % units), pass = (int)(i / ((size_t)65 * 128 * units));
        const int bh = u / G, g = u % G;
        float a = 0.f;
        for (int sp = 0; sp < nsplit; ++sp)
            a += part[(((size_t)pass * units * nsplit + ((size_t)bh * nsplit + sp) * G + g) * 128 +
                       row) * 80 + col];
        total[(((size_t)pass * units + u) * 128 + row) * 80 + col] = a;
    }
}

// Chunk splits per (pass, sequence, group) for the non-causal modes: enough CTAs for a few
// waves of ~152 SMs, every split non-empty (depends on the shape only, so the workspace size
// is known before the call).
int nc_splits(const Problem& p)
{
    const int units = p.B * p.H * (p.M / 64), nch = (p.N + kC - 1) / kC;
    const int target = std::max(1, std::min(nch, (4 * 152 + 2 * units - 1) / (2 * units)));
    const int cps = (nch + target - 1) / target;
    return (nch + cps - 1) / cps;
}

// Scratch layout (every region 256-byte aligned): dW partials [2 half][128][64], key
// weights [B*H*N] (prefactor), dtau partials [2 half]; non-causal also partial states
// [2 half][128][80] and totals [2 units][128][80] (half = B*H*G*nsplit, units = B*H*G).
struct BwdWs {
    size_t part, kw, dtau, state_part, state_total, total;
};
BwdWs bwd_ws(const Problem& p)
{
    const size_t units = (size_t)p.B * p.H * (p.M / 64);
    const size_t half = units * (p.causal ? 1 : nc_splits(p));
    auto a64 = [](size_t n) { return align_up(n, 64); };  // floats
    BwdWs w;
    w.part = 0;
    w.kw = a64(w.part + 2 * half * 128 * 64);
    w.dtau = a64(w.kw + (size_t)p.B * p.H * p.N);
    w.state_part = a64(w.dtau + 2 * half);
    w.state_total = a64(w.state_part + (p.causal ? 0 : 2 * half * 128 * 80));
    w.total = a64(w.state_total + (p.causal ? 0 : 2 * units * 128 * 80));
    return w;  // in floats
}

struct BwdArgs {
    CUtensorMap mq, mk, mv, mdo, mo;
};

// One launch of tc_bwd_kernel<NS, KW, CS, MODE>: 2 * units * nsplit CTAs, clusters of CS.
template <bool NS, bool KW, int CS, int MODE>
cudaError_t launch_mode(const Problem& p, const BwdArgs& m, const void* q, const void* k,
                        const void* v, const float* W1, const float* W2, const float* tau,
                        const void* out, const float* den, const void* dout, void* dq, void* dk,
                        void* dv, float* f, const BwdWs& w, int nsplit, int* status,
                        cudaStream_t s)
{
    const int smem = (int)BwCfg<NS>::BYTES + 1024;
    auto kb = tc_bwd_kernel<NS, KW, CS, MODE>;
    cudaError_t e = cudaFuncSetAttribute(kb, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    typedef const __nv_bfloat16* CB;
    typedef __nv_bfloat16* B16;
    const int units = p.B * p.H * (p.M / 64);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(2 * units * nsplit));
    cfg.blockDim = dim3(kThreadsB);
    cfg.dynamicSmemBytes = (size_t)smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;  // the frequency groups of one (pass, sequence, split)
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kb, m.mq, m.mk, m.mv, m.mdo, m.mo, p.H, p.N, p.M, p.M / 64,
                              p.causal, (CB)q, (CB)k, (CB)v, W1, W2, (CB)out, den, (CB)dout,
                              (B16)dq, (B16)dk, (B16)dv, f + w.part, KW ? f + w.kw : nullptr, tau,
                              f + w.dtau, units, nsplit, f + w.state_part,
                              (const float*)(f + w.state_total), status);
}

template <bool NS, bool KW>
cudaError_t launch_bwd(const Problem& p, const void* q, const void* k, const void* v,
                       const float* W1, const float* W2, const float* tau, const void* out,
                       const float* den, const void* dout, void* dq, void* dk, void* dv,
                       float* dW1, float* dW2, float* dtau, void* scratch, int* status,
                       cudaStream_t s)
{
    const int BH = p.B * p.H, G = p.M / 64;
    float* f = static_cast<float*>(scratch);
    const BwdWs w = bwd_ws(p);
    cudaError_t e = cudaSuccess;
    if (KW && (e = launch_key_weights(p, k, tau, f + w.kw, s)) != cudaSuccess) return e;
    BwdArgs m;
    if (!make_act_map(&m.mq, q, BH, p.N) || !make_act_map(&m.mk, k, BH, p.N) ||
        !make_act_map(&m.mv, v, BH, p.N) || !make_act_map(&m.mdo, dout, BH, p.N) ||
        !make_act_map(&m.mo, out, BH, p.N))
        return cudaErrorInvalidValue;
    int nsplit = 1;
    if (p.causal) {
        e = G == 2 ? launch_mode<NS, KW, 2, kCausal>(p, m, q, k, v, W1, W2, tau, out, den, dout, dq,
                                                     dk, dv, f, w, 1, status, s)
                   : launch_mode<NS, KW, 1, kCausal>(p, m, q, k, v, W1, W2, tau, out, den, dout, dq,
                                                     dk, dv, f, w, 1, status, s);
        if (e != cudaSuccess) return e;
    } else {
        nsplit = nc_splits(p);
        e = launch_mode<NS, KW, 1, kState>(p, m, q, k, v, W1, W2, tau, out, den, dout, dq, dk, dv,
                                           f, w, nsplit, status, s);
        if (e != cudaSuccess) return e;
        const int units = BH * G;
        nc_state_reduce_kernel<<<152 * 4, 256, 0, s>>>(units, G, nsplit, f + w.state_part,
                                                       f + w.state_total);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        e = G == 2 ? launch_mode<NS, KW, 2, kGrad>(p, m, q, k, v, W1, W2, tau, out, den, dout, dq,
                                                   dk, dv, f, w, nsplit, status, s)
                   : launch_mode<NS, KW, 1, kGrad>(p, m, q, k, v, W1, W2, tau, out, den, dout, dq,
                                                   dk, dv, f, w, nsplit, status, s);
        if (e != cudaSuccess) return e;
    }
    const size_t work = (size_t)p.H * p.M * 64;
    tc_dw_reduce_kernel<<<(int)std::min<size_t>((work + 255) / 256, 152 * 8), 256, 0, s>>>(
        p.B, p.H, p.M, G, nsplit, p.nonstat, f + w.part, dW1, dW2, f + w.dtau,
        KW ? dtau : nullptr);
    return cudaGetLastError();
}

}  // namespace

// bf16, d = 64, M in {64, 128}: causal (two scans) and non-causal (totals, then every
// chunk independently).
bool tc_bwd_supported(const Problem& p)
{
    return p.bf16 && p.d == 64 && (p.M == 64 || p.M == 128);
}

int tc_bwd_launches(const Problem& p, bool tau)
{
    return (p.causal ? 2 : 4) + (tau ? 1 : 0);
}

size_t tc_bwd_ws_bytes(const Problem& p) { return bwd_ws(p).total * sizeof(float); }

cudaError_t launch_tc_bwd(const Problem& p, const void* q, const void* k, const void* v,
                          const float* W1, const float* W2, const float* tau, const void* out,
                          const float* den, const void* dout, void* dq, void* dk, void* dv,
                          float* dW1, float* dW2, float* dtau, void* scratch, int* status,
                          cudaStream_t s)
{
#define FLEX_BWD_ARGS p, q, k, v, W1, W2, tau, out, den, dout, dq, dk, dv, dW1, dW2, dtau, scratch, status, s
    if (p.nonstat)
        return tau ? launch_bwd<true, true>(FLEX_BWD_ARGS) : launch_bwd<true, false>(FLEX_BWD_ARGS);
    return tau ? launch_bwd<false, true>(FLEX_BWD_ARGS) : launch_bwd<false, false>(FLEX_BWD_ARGS);
#undef FLEX_BWD_ARGS
}

}  // namespace flex
