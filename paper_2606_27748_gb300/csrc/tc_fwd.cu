// Causal forward of RFF linear attention on the 5th-generation tensor cores (tcgen05).
//
// Chunked scan of Eq. (linear att) with j <= i: the sequence is cut into chunks of 128
// tokens; inside a chunk the masked kernel matrix A = phi(Q) phi(K)^T is applied directly
// (A V), across chunks the running state S = sum phi(k) v^T and z = sum phi(k) carries the
// prefix (phi(Q) S, phi(Q) z).  phi never leaves the SM: the projection x W^T lands in
// tensor memory, the CUDA cores turn it into cos/sin features (Eq. phi_n, or the product
// form of Eq. phi_non) and write them as bf16 MMA operands to shared memory.
//
// Features are processed in groups of 64 frequencies (128 features: 64 cos + 64 sin); A,
// phi(Q) S and phi(Q) z accumulate over the groups, S and z are held per group.  Features
// are unscaled ([cos, sin] instead of M^{-1/2}[cos, sin]): the factor cancels in the
// output, and only the stored denominator is rescaled (den = den' / M).
//
// Warp roles (608 threads), handshakes on mbarriers:
//   warp 0      TMA: q, k, v chunk tiles (128B swizzle) into shared memory
//   warp 1      one thread issues the attention MMAs (QK, numerator, state, A V); owns the
//               tensor-memory allocation
//   warp 18     one thread issues the projection MMAs.  A thread that issues an MMA blocks
//               while the tensor core's queue is full, so projections get their own issuer
//               and never wait behind a long attention step
//   warps 2-9   features: projection (TMEM) -> cos/sin -> bf16 phi tiles (shared memory);
//               warps 2-5 take frequencies 0-31 of a group, warps 6-9 frequencies 32-63
//   warps 10-17 epilogue, two halves of 4 warps: causal mask + bf16 of A (written back
//               into TMEM as the A operand of A V), output rows, bf16 snapshot of S and z
//               for the next chunk; each half takes half of the columns (or one group)
//
// Sequence split: when there are SMs to spare, a sequence is cut into `splits` segments
// handled by different CTAs with no waiting between them: the CTA of segment j first runs
// a k-only pass over the chunks before its segment (projection + features of k and the
// state update, no outputs) to build the state prefix, then its own chunks.  Segment
// lengths halve from one segment to the next, which balances the work because a k-only
// chunk costs about half a full chunk.
//
// z rides in S as an extra column: the state update multiplies phi(K)^T by [V | 1], and
// the output MMAs multiply by [S | z] and [V | 1], so column 64 of the output accumulator
// is the denominator, built from exactly the bf16 values that build the numerator.
//
// Tensor memory (512 columns x 128 lanes, fp32):
//   [0,128)    projection of one group (s: 64 cols a; n: 64 cols u, 64 cols w)
//   [128,256)  A = phi(Q) phi(K)^T (row = query, col = key); after the epilogue, columns
//              [0,32) and [64,96) hold bf16(masked A) of keys 0-63 and 64-127, two per column
//   [256,336)  phi(Q) [S | z] + A [V | 1]: numerator in 0-63, denominator in 64
//   [336,336+80G)  [S | z] per group (lane = feature), z in column 64 of each
#include <cuda.h>

#include "flex_internal.h"
#include "tc_common.cuh"
#include "tc_util.cuh"

namespace flex {
namespace {
using namespace tc;

constexpr int kC = 128;            // tokens per chunk = MMA M
constexpr int kThreadsTC = 608;    // 19 warps
constexpr int kWarpTMA = 0, kWarpMMA = 1, kWarpFW = 2, kWarpEW = 10, kEpiWarps = 8;
constexpr int kWarpProj = 18;

template <bool NS, int G>
struct Cfg {
    static constexpr int P = NS ? 128 : 64;  // projection columns per group
    // shared memory offsets (bytes, 1024-aligned); X0/X1 hold q/k tiles.  VONE is the
    // second 64-column block of [V | 1] (column 0 = 1, the rest 0), reached from either V
    // buffer through the descriptor's leading byte offset.
    static constexpr uint32_t X0 = 0, X1 = 16384, V0 = 32768, V1 = 49152, VONE = 65536;
    static constexpr uint32_t W = 81920;
    static constexpr uint32_t PQ = W + G * P * 128;
    static constexpr uint32_t PK = PQ + 32768;
    // [S | z] snapshot per group, K-major: 80 rows (64 dcols, z, 15 zero rows) x 128
    // features = two 64-feature blocks of 80 x 128 bytes
    static constexpr uint32_t SX = PK + 32768;
    static constexpr uint32_t SX_BLOCK = 80 * 128, SX_GROUP = 2 * SX_BLOCK;
    static constexpr uint32_t BYTES = SX + G * SX_GROUP;
    // tensor memory columns
    static constexpr uint32_t T_P = 0, T_A = 128, T_O = 256, T_S = 336;
    static_assert(T_S + 80 * G <= 512, "tensor memory budget");
    static_assert(BYTES + 1024 <= 232448, "shared memory budget");
};

struct Bars {
    uint64_t x_full[2], x_free[2], v_full[2], v_free[2];
    uint64_t p_full, p_free, phiq_full, phik_full, phiq_free, phik_free;
    uint64_t attn_done, a_ready, o_ready, epi_done;
};

// First chunk of segment j of `splits` (lengths proportional to 2^-j), rounded.
__device__ __forceinline__ int segment_bound(int nch, int splits, int j)
{
    const long long den = (1LL << splits) - 1;
    const long long num = (long long)nch * ((1LL << splits) - (1LL << (splits - j)));
    return (int)((2 * num + den) / (2 * den));
}

template <bool NS, int G>
__global__ void __maxnreg__(96)
    tc_fwd_causal_kernel(const __grid_constant__ CUtensorMap tmap_q,
                         const __grid_constant__ CUtensorMap tmap_k,
                         const __grid_constant__ CUtensorMap tmap_v, int H, int N, int M,
                         int splits, const float* __restrict__ W1,
                         const float* __restrict__ W2, __nv_bfloat16* __restrict__ out,
                         float* __restrict__ den, int* status)
{
    using L = Cfg<NS, G>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sb = smem_u32(sm);
    __shared__ Bars bars;
    __shared__ uint32_t tmem_base_sh;
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.x / splits, seg = blockIdx.x % splits, h = bh % H;
    const int nch = (N + kC - 1) / kC;
    const int cb = segment_bound(nch, splits, seg), ce = segment_bound(nch, splits, seg + 1);
    if (cb >= ce) return;  // uniform over the CTA
    const size_t base = (size_t)bh * N * 64;

    // ---- set-up: frequencies (bf16, K-major rows), ones, zero state snapshots ----
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
    for (int idx = tid; idx < 16384 / 16; idx += kThreadsTC)  // [1, 0, ..., 0] rows
        st_shared_v4(sb + L::VONE + idx * 16, 0, 0, 0, 0);
    for (int idx = tid; idx < G * L::SX_GROUP / 16; idx += kThreadsTC)
        st_shared_v4(sb + L::SX + idx * 16, 0, 0, 0, 0);
    __syncthreads();
    for (int r = tid; r < kC; r += kThreadsTC)
        *reinterpret_cast<uint16_t*>(sm + L::VONE + swz128(r, 0)) = 0x3F80u;  // bf16 1.0
    if (tid == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars.x_full[i], 1);
            mbar_init(&bars.x_free[i], 1);
            mbar_init(&bars.v_full[i], 1);
            mbar_init(&bars.v_free[i], 1);
        }
        mbar_init(&bars.p_full, 1);
        mbar_init(&bars.p_free, 8);
        mbar_init(&bars.phiq_full, 8);
        mbar_init(&bars.phik_full, 8);
        mbar_init(&bars.phiq_free, 1);
        mbar_init(&bars.phik_free, 1);
        mbar_init(&bars.attn_done, 1);
        mbar_init(&bars.a_ready, kEpiWarps);
        mbar_init(&bars.o_ready, 1);
        mbar_init(&bars.epi_done, kEpiWarps);
        abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == kWarpMMA) {
        tmem_alloc(&tmem_base_sh, 512);
        tmem_relinquish();
    }
    fence_proxy_async();
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tm = tmem_base_sh;

    if (warp == kWarpTMA) {
        // ================= TMA producer =================
        // Main chunks: q -> X0, k -> X1.  k-only prefix chunks alternate k between X1 and
        // X0, so the next tile loads while the current one is projected.
        if (lane == 0) {
            uint32_t ph_xfree[2] = {0, 0}, ph_vfree[2] = {0, 0};
            bool used_x[2] = {false, false}, used_v[2] = {false, false};
            auto load = [&](int b, const CUtensorMap* map, int t0) -> bool {
                if (used_x[b]) {
                    if (!bar_wait(&bars.x_free[b], ph_xfree[b], &abort_flag, status)) return false;
                    ph_xfree[b] ^= 1;
                }
                used_x[b] = true;
                mbar_arrive_expect_tx(&bars.x_full[b], kTileBytes);
                tma_load_3d(sb + (b ? L::X1 : L::X0), map, 0, t0, bh, &bars.x_full[b]);
                return true;
            };
            for (int c = 0; c < ce; ++c) {
                const int t0 = c * kC;
                if (c + 1 < ce) {  // the next chunk's tiles into L2 while this one is used
                    if (c + 1 >= cb) tma_prefetch_3d(&tmap_q, 0, t0 + kC, bh);
                    tma_prefetch_3d(&tmap_k, 0, t0 + kC, bh);
                    tma_prefetch_3d(&tmap_v, 0, t0 + kC, bh);
                }
                if (c >= cb) {
                    if (!load(0, &tmap_q, t0) || !load(1, &tmap_k, t0)) break;
                } else {
                    if (!load((c & 1) ? 0 : 1, &tmap_k, t0)) break;
                }
                const int vb = c & 1;
                if (used_v[vb]) {
                    if (!bar_wait(&bars.v_free[vb], ph_vfree[vb], &abort_flag, status)) break;
                    ph_vfree[vb] ^= 1;
                }
                used_v[vb] = true;
                mbar_arrive_expect_tx(&bars.v_full[vb], kTileBytes);
                tma_load_3d(sb + (vb ? L::V1 : L::V0), &tmap_v, 0, t0, bh, &bars.v_full[vb]);
            }
        }
    } else if (warp == kWarpMMA || warp == kWarpProj) {
        // ================= MMA issue (one thread per role) =================
        if (lane == 0) {
            constexpr uint32_t I_PROJ = idesc_bf16(128, L::P, 0, 0);
            constexpr uint32_t I_QK = idesc_bf16(128, 128, 0, 0);
            constexpr uint32_t I_QS = idesc_bf16(128, 80, 0, 0);
            constexpr uint32_t I_KV = idesc_bf16(128, 80, 1, 1);
            constexpr uint32_t I_AV = idesc_bf16(128, 80, 0, 1);
            bool ok = true;
            auto wait = [&](uint64_t* bar, uint32_t& ph) {
                if (!ok) return;
                ok = bar_wait(bar, ph, &abort_flag, status);
                ph ^= 1;
            };
            // Descriptors are built once; an operand K step adds its byte offset / 16 to
            // the start-address field (addresses stay below 256 KB: no carry out).
            auto adv = [](uint64_t d, uint32_t bytes) { return d + (bytes >> 4); };
            if (warp == kWarpProj) {
                // projections: per chunk, per group, q (main chunks) then k
                const uint64_t d_x[2] = {sdesc(sb + L::X0, 16, 1024), sdesc(sb + L::X1, 16, 1024)};
                const uint64_t d_w = sdesc(sb + L::W, 16, 1024);
                uint32_t ph_xfull[2] = {0, 0}, ph_pfree = 0;
                int nproj = 0;
                for (int c = 0; c < ce && ok; ++c) {
                    const bool main = c >= cb;
                    for (int g = 0; g < G && ok; ++g) {
                        for (int which = main ? 0 : 1; which < 2 && ok; ++which) {
                            const int buf = which == 0 ? 0 : (main ? 1 : ((c & 1) ? 0 : 1));
                            if (g == 0) wait(&bars.x_full[buf], ph_xfull[buf]);
                            if (nproj > 0) wait(&bars.p_free, ph_pfree);
                            if (!ok) break;
                            fence_after_sync();
                            const uint64_t wd = adv(d_w, g * L::P * 128);
#pragma unroll
                            for (int ks = 0; ks < 4; ++ks)
                                mma_bf16(tm + L::T_P, adv(d_x[buf], ks * 32), adv(wd, ks * 32),
                                         I_PROJ, ks > 0);
                            mma_commit(&bars.p_full);
                            if (g == G - 1) mma_commit(&bars.x_free[buf]);
                            ++nproj;
                        }
                    }
                }
            } else {
                // attention MMAs of each group, then A V of each main chunk
                const uint64_t d_pq = sdesc(sb + L::PQ, 16, 1024);
                const uint64_t d_pk = sdesc(sb + L::PK, 16, 1024);
                const uint64_t d_pk_mn = sdesc(sb + L::PK, 16384, 1024);
                const uint64_t d_sx = sdesc(sb + L::SX, 16, 1024);
                const uint64_t d_v[2] = {sdesc(sb + L::V0, L::VONE - L::V0, 1024),
                                         sdesc(sb + L::V1, L::VONE - L::V1, 1024)};
                uint32_t ph_vfull[2] = {0, 0};
                uint32_t ph_phiq = 0, ph_phik = 0, ph_aready = 0, ph_epi = 0;
                for (int c = 0; c < ce && ok; ++c) {
                    const bool main = c >= cb;
                    const uint64_t vd = d_v[c & 1];
                    for (int g = 0; g < G && ok; ++g) {
                        if (main) wait(&bars.phiq_full, ph_phiq);
                        wait(&bars.phik_full, ph_phik);
                        if (g == 0) {
                            wait(&bars.v_full[c & 1], ph_vfull[c & 1]);
                            if (main) wait(&bars.epi_done, ph_epi);
                        }
                        if (!ok) break;
                        fence_after_sync();
                        if (main) {
                            const uint64_t sxd = adv(d_sx, g * L::SX_GROUP);
#pragma unroll
                            for (int ks = 0; ks < 8; ++ks) {  // K = 128 features of group g
                                const uint32_t kofs = (ks >> 2) * 16384 + (ks & 3) * 32;
                                const uint64_t aq = adv(d_pq, kofs);
                                const uint32_t acc = (g > 0 || ks > 0) ? 1u : 0u;
                                mma_bf16(tm + L::T_A, aq, adv(d_pk, kofs), I_QK, acc);
                                mma_bf16(tm + L::T_O, aq,
                                         adv(sxd, (ks >> 2) * L::SX_BLOCK + (ks & 3) * 32), I_QS,
                                         acc);
                            }
                            mma_commit(&bars.phiq_free);  // phi(Q) no longer read
                        }
                        const uint32_t acc_s = c > 0 ? 1u : 0u;
#pragma unroll
                        for (int ks = 0; ks < 8; ++ks)  // K = 128 tokens of the chunk
                            mma_bf16(tm + L::T_S + 80 * g, adv(d_pk_mn, ks * 2048),
                                     adv(vd, ks * 2048), I_KV, (acc_s | (ks > 0)) ? 1u : 0u);
                        mma_commit(&bars.phik_free);  // phi(K) no longer read
                        if (g == G - 1) {
                            if (main || c == cb - 1) mma_commit(&bars.attn_done);
                            if (!main) mma_commit(&bars.v_free[c & 1]);
                        }
                    }
                    if (main && ok) {
                        wait(&bars.a_ready, ph_aready);
                        if (!ok) break;
                        fence_after_sync();
#pragma unroll
                        for (int ks = 0; ks < 8; ++ks)  // keys 16ks..16ks+15: bf16 A columns
                            mma_bf16_tmem_a(tm + L::T_O, tm + L::T_A + 64 * (ks >> 2) + 8 * (ks & 3),
                                            adv(vd, ks * 2048), I_AV, 1u);
                        mma_commit(&bars.o_ready);
                        mma_commit(&bars.v_free[c & 1]);
                    }
                }
            }
        }
    } else if (warp < kWarpEW) {
        // ================= features =================
        const int half = (warp - kWarpFW) >> 2, quad = warp & 3, t = 32 * quad + lane;
        const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16) + L::T_P;
        uint32_t ph_pfull = 0;
        int n = 0, nq = 0;  // groups processed so far (all / main chunks)
        for (int c = 0; c < ce; ++c) {
            const bool main = c >= cb;
            const bool valid = t < min(kC, N - c * kC);
            for (int g = 0; g < G; ++g, ++n, nq += main ? 1 : 0) {
                for (int which = main ? 0 : 1; which < 2; ++which) {  // 0: q, 1: k
                    if (!bar_wait(&bars.p_full, ph_pfull, &abort_flag, status)) goto fw_out;
                    ph_pfull ^= 1;
                    fence_after_sync();
                    float a[32], w[32];
                    tmem_ld16(tm_row + 32 * half, *reinterpret_cast<float(*)[16]>(&a[0]));
                    tmem_ld16(tm_row + 32 * half + 16, *reinterpret_cast<float(*)[16]>(&a[16]));
                    if (NS) {
                        tmem_ld16(tm_row + 64 + 32 * half, *reinterpret_cast<float(*)[16]>(&w[0]));
                        tmem_ld16(tm_row + 64 + 32 * half + 16,
                                  *reinterpret_cast<float(*)[16]>(&w[16]));
                    }
                    tmem_wait_ld();
                    fence_before_sync();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&bars.p_free);
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
                    // the tile is free once the previous group's MMAs that read it are done
                    if (which == 0 ? (nq > 0 && !bar_wait(&bars.phiq_free, (nq - 1) & 1,
                                                          &abort_flag, status))
                                   : (n > 0 && !bar_wait(&bars.phik_free, (n - 1) & 1,
                                                         &abort_flag, status)))
                        goto fw_out;
                    const uint32_t dst = sb + (which ? L::PK : L::PQ);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const uint32_t off = swz128(t, (4 * half + j) * 8);
                        st_shared_v4(dst + off, pc[4 * j], pc[4 * j + 1], pc[4 * j + 2],
                                     pc[4 * j + 3]);
                        st_shared_v4(dst + 16384 + off, ps[4 * j], ps[4 * j + 1], ps[4 * j + 2],
                                     ps[4 * j + 3]);
                    }
                    fence_proxy_async();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(which ? &bars.phik_full : &bars.phiq_full);
                }
            }
        }
    fw_out:;
    } else {
        // ================= epilogue =================
        // Two halves of 4 warps (one warp per lane quadrant each): half eh takes keys
        // [64eh, 64eh+64) of A, output columns [32eh, 32eh+32), and group eh of the state
        // (G = 2) or its state columns [32eh, 32eh+32) (G = 1).
        const int eh = (warp - kWarpEW) >> 2, quad = warp & 3, t = 32 * quad + lane;
        const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);
        uint32_t ph_attn = 0, ph_o = 0;
        auto snapshot = [&]() {
            // K-major [S | z]: row e holds S[f][e] over the features f of one group
            constexpr int NCOL = G == 2 ? 64 : 32;
            const int g = G == 2 ? eh : 0, e0 = G == 2 ? 0 : 32 * eh;
            float s_[NCOL];
#pragma unroll
            for (int j = 0; j < NCOL / 16; ++j)
                tmem_ld16(tm_row + L::T_S + 80 * g + e0 + 16 * j,
                          *reinterpret_cast<float(*)[16]>(&s_[16 * j]));
            float zz[16];
            const bool with_z = G == 2 || eh == 0;
            if (with_z) tmem_ld16(tm_row + L::T_S + 80 * g + 64, zz);
            tmem_wait_ld();
            uint8_t* blk = sm + L::SX + g * L::SX_GROUP + (t >> 6) * L::SX_BLOCK;
            const uint32_t col = t & 63;
#pragma unroll
            for (int e = 0; e < NCOL; ++e)
                *reinterpret_cast<__nv_bfloat16*>(blk + swz128(e0 + e, col)) =
                    __float2bfloat16_rn(s_[e]);
            if (with_z)
                *reinterpret_cast<__nv_bfloat16*>(blk + swz128(64, col)) =
                    __float2bfloat16_rn(zz[0]);
        };
        auto signal = [&](uint64_t* bar) {
            fence_proxy_async();
            fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar);
        };
        if (cb > 0) {  // the k-only prefix ends here: snapshot its state
            if (!bar_wait(&bars.attn_done, ph_attn, &abort_flag, status)) goto ew_out;
            ph_attn ^= 1;
            fence_after_sync();
            snapshot();
        }
        signal(&bars.epi_done);
        for (int c = cb; c < ce; ++c) {
            const int t0 = c * kC;
            const bool valid = t < min(kC, N - t0);
            if (!bar_wait(&bars.attn_done, ph_attn, &abort_flag, status)) goto ew_out;
            ph_attn ^= 1;
            fence_after_sync();
            // causal mask + bf16; keys 32b..32b+31 of this half (columns 64eh + 32b ..) go
            // to columns 64eh + 16b .., which this thread has already read
#pragma unroll
            for (int b = 0; b < 2; ++b) {
                const uint32_t col = L::T_A + 64 * eh + 32 * b;
                float a[32];
                tmem_ld16(tm_row + col, *reinterpret_cast<float(*)[16]>(&a[0]));
                tmem_ld16(tm_row + col + 16, *reinterpret_cast<float(*)[16]>(&a[16]));
                tmem_wait_ld();
                uint32_t pk2[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const int j0 = 64 * eh + 32 * b + 2 * i;
                    pk2[i] = pack_bf16(j0 <= t ? a[2 * i] : 0.f, j0 + 1 <= t ? a[2 * i + 1] : 0.f);
                }
                tmem_st16(tm_row + L::T_A + 64 * eh + 16 * b, pk2);
            }
            tmem_wait_st();
            signal(&bars.a_ready);

            if (!bar_wait(&bars.o_ready, ph_o, &abort_flag, status)) goto ew_out;
            ph_o ^= 1;
            fence_after_sync();
            float o[32], dn[16];
            tmem_ld16(tm_row + L::T_O + 32 * eh, *reinterpret_cast<float(*)[16]>(&o[0]));
            tmem_ld16(tm_row + L::T_O + 32 * eh + 16, *reinterpret_cast<float(*)[16]>(&o[16]));
            tmem_ld16(tm_row + L::T_O + 64, dn);
            tmem_wait_ld();
            if (valid) {
                const float inv = 1.f / dn[0];
                uint4* dst = reinterpret_cast<uint4*>(out + base + (size_t)(t0 + t) * 64 + 32 * eh);
#pragma unroll
                for (int cc = 0; cc < 4; ++cc)
                    dst[cc] = make_uint4(pack_bf16(o[8 * cc] * inv, o[8 * cc + 1] * inv),
                                         pack_bf16(o[8 * cc + 2] * inv, o[8 * cc + 3] * inv),
                                         pack_bf16(o[8 * cc + 4] * inv, o[8 * cc + 5] * inv),
                                         pack_bf16(o[8 * cc + 6] * inv, o[8 * cc + 7] * inv));
                if (den && eh == 0) den[(size_t)bh * N + t0 + t] = dn[0] / (float)M;
            }
            if (c + 1 < ce) snapshot();
            signal(&bars.epi_done);
        }
    ew_out:;
    }

    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == kWarpMMA) tmem_dealloc(tm, 512);
}

template <bool NS, int G>
cudaError_t launch_one(const Problem& p, const void* q, const void* k, const void* v,
                       const float* W1, const float* W2, void* out, float* den, int* status,
                       cudaStream_t s)
{
    CUtensorMap mq, mk, mv;
    const int BH = p.B * p.H;
    if (!make_act_map(&mq, q, BH, p.N) || !make_act_map(&mk, k, BH, p.N) ||
        !make_act_map(&mv, v, BH, p.N))
        return cudaErrorInvalidValue;
    const int splits = tc_fwd_splits(p, sm_count());
    auto kern = tc_fwd_causal_kernel<NS, G>;
    const int smem = (int)Cfg<NS, G>::BYTES + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    kern<<<BH * splits, kThreadsTC, smem, s>>>(mq, mk, mv, p.H, p.N, p.M, splits, W1, W2,
                                               (__nv_bfloat16*)out, den, status);
    return cudaGetLastError();
}

}  // namespace

int tc_fwd_splits(const Problem& p, int sms)
{
    const long long BH = (long long)p.B * p.H;
    const int nch = (p.N + kC - 1) / kC;
    if (sms > 0 && 3 * BH <= sms && nch >= 14) return 3;
    if (sms > 0 && 2 * BH <= sms && nch >= 6) return 2;
    return 1;
}

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
