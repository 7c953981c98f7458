// Non-causal forward of RFF linear attention on the tensor cores (tcgen05).
//
// Eq. (linear att) with sums over all j: S = sum_j phi(k_j) v_j^T and z = sum_j phi(k_j)
// are shared by every query ("precomputed and shared across all positional queries",
// Sec. 2.2), so the work splits in two phases that both parallelise over the sequence:
//
//   1. state:  every (b, h, split) unit runs over its chunks of 128 tokens: projection of
//              k (TMEM) -> cos/sin features (CUDA cores, bf16 in shared memory) ->
//              [S | z]_part += phi(K)^T [V | 1] (TMEM), then writes its partial in fp32;
//   2. reduce: the partials of a sequence are summed in a fixed order (deterministic);
//   3. output: every unit loads the total as a bf16 operand and runs over its chunks:
//              projection of q -> features -> phi(Q) [S | z] (TMEM) -> out = num / den.
//
// z rides as column 64 of [S | z]: the state MMA multiplies by [V | 1] (a constant ones
// block reached through the descriptor's leading byte offset) and the output MMA by the
// K-major [S | z] snapshot, so the denominator comes out as column 64 of the output.
// Features are unscaled (the M^{-1/2} of Eq. phi_n / phi_non cancels); den = den' / M.
//
// Warp roles (736 threads): warp 0 TMA of the q or k tiles, warp 1 issues the projection
// MMAs, warp 22 the state (or output) MMAs, warps 2-17 features (four per lane quadrant,
// warp 2 + 4 fq + r' taking frequencies 16 fq .. 16 fq + 15 of a group), warps 18-21
// epilogue (state mode: warp 21 first issues the v tiles' TMA; output mode: rows staged in
// shared memory and written by TMA stores).  Projection buffers (TMEM) and feature tiles
// (shared memory) are double-buffered, so the feature warps compute job j+1 while the
// tensor core consumes job j.
#include <cuda.h>

#include <algorithm>

#include "flex_internal.h"
#include "tc_common.cuh"
#include "tc_util.cuh"

namespace flex {
namespace {
using namespace tc;

constexpr int kC = 128;
constexpr int kThreadsNC = 736;  // 23 warps
constexpr int kWarpTMA = 0, kWarpMMA = 1, kWarpFW = 2, kNumFW = 16, kWarpEW = 18, kWarpCons = 22;
constexpr int kAhead = 4;  // chunks prefetched into L2 ahead of their tile load
constexpr int kSMs = 152;
constexpr int kTargetUnits = 8 * kSMs;  // most work units per launch
constexpr int kSetupChunks = 5;         // fixed cost of a unit, in chunk times

enum { kState = 0, kOut = 1 };

template <bool NS, int G>
struct NcCfg {
    static constexpr int P = NS ? 128 : 64;
    static constexpr uint32_t X0 = 0, X1 = 16384, V0 = 32768, V1 = 49152, VONE = 65536;
    static constexpr uint32_t W = 81920;
    static constexpr uint32_t PB0 = W + G * P * 128, PB1 = PB0 + 32768;
    static constexpr uint32_t SX = PB1 + 32768;
    static constexpr uint32_t SX_BLOCK = 80 * 128, SX_GROUP = 2 * SX_BLOCK;
    static constexpr uint32_t BYTES = SX + G * SX_GROUP;
    static constexpr uint32_t T_P0 = 0, T_P1 = 128, T_S = 256, T_O0 = 256, T_O1 = 336;
    static_assert(T_S + 80 * G <= 512 && T_O1 + 80 <= 512, "tensor memory budget");
    static_assert(BYTES + 1024 <= 232448, "shared memory budget");
};

struct NcBars {
    uint64_t x_full[2], x_free[2], v_full[2], v_free[2];
    uint64_t p_full[2], p_free[2], phi_full[2], phi_free[2];
    uint64_t o_full[2], o_free[2], state_done;
};

// partial / total [S | z] rows: [unit][group][feature 128][80 floats]
constexpr int kRow = 80;

// KW: key weights of the norm prefactor given (compile-time; the plain kernel is unchanged)
template <int MODE, bool NS, int G, bool KW>
__global__ void __launch_bounds__(kThreadsNC, 1)
    tc_nc_kernel(const __grid_constant__ CUtensorMap tmap_x,
                 const __grid_constant__ CUtensorMap tmap_v, int H, int N, int M, int splits,
                 const float* __restrict__ W1, const float* __restrict__ W2,
                 const float* __restrict__ kw, float* __restrict__ part,
                 const float* __restrict__ total, __nv_bfloat16* __restrict__ out,
                 float* __restrict__ den, int* status)
{
    using L = NcCfg<NS, G>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sb = smem_u32(sm);
    __shared__ NcBars bars;
    __shared__ uint32_t tmem_base_sh;
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.x / splits, sp = blockIdx.x % splits, h = bh % H;
    const int nch = (N + kC - 1) / kC;
    const int c0 = (int)((long long)sp * nch / splits), c1 = (int)((long long)(sp + 1) * nch / splits);
    const int nc = c1 - c0;  // chunks of this unit (>= 1: splits <= nch)

    // ---- set-up: frequencies, [V | 1] ones block, [S | z] snapshot (output phase) ----
    for (int idx = tid; idx < G * L::P * 8; idx += kThreadsNC) {
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
    if (MODE == kState) {
        for (int idx = tid; idx < 16384 / 16; idx += kThreadsNC)
            st_shared_v4(sb + L::VONE + idx * 16, 0, 0, 0, 0);
        __syncthreads();
        for (int r = tid; r < kC; r += kThreadsNC)
            *reinterpret_cast<uint16_t*>(sm + L::VONE + swz128(r, 0)) = 0x3F80u;  // 1.0
    } else {
        // K-major [S | z]: row e (dcol e, z at 64, zero rows 65-79) over features f
        const float* tot = total + (size_t)bh * G * 128 * kRow;
        for (int idx = tid; idx < G * 128 * 80; idx += kThreadsNC) {
            const int g = idx / (128 * 80), rem = idx % (128 * 80);
            const int e = rem / 128, f = rem % 128;
            const float val = e <= 64 ? tot[((size_t)g * 128 + f) * kRow + e] : 0.f;
            *reinterpret_cast<__nv_bfloat16*>(sm + L::SX + g * L::SX_GROUP + (f >> 6) * L::SX_BLOCK +
                                              swz128(e, f & 63)) = __float2bfloat16_rn(val);
        }
    }
    if (tid == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars.x_full[i], 1);
            mbar_init(&bars.x_free[i], 1);
            mbar_init(&bars.v_full[i], 1);
            mbar_init(&bars.v_free[i], 1);
            mbar_init(&bars.p_full[i], 1);
            mbar_init(&bars.p_free[i], kNumFW);
            mbar_init(&bars.phi_full[i], kNumFW);
            mbar_init(&bars.phi_free[i], 1);
            mbar_init(&bars.o_full[i], 1);
            mbar_init(&bars.o_free[i], 4);
        }
        mbar_init(&bars.state_done, 1);
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
    const int njobs = nc * G;

    if (warp == kWarpTMA) {
        // q or k tiles (v has its own thread: a v buffer frees late, after the state MMA two
        // chunks back, and must not hold up the next projection's tile)
        if (lane == 0) {
            uint32_t ph_x[2] = {0, 0};
            for (int i = 0; i < nc; ++i) {
                const int b = i & 1, t0 = (c0 + i) * kC;
                if (i + kAhead < nc) tma_prefetch_3d(&tmap_x, 0, t0 + kAhead * kC, bh);  // into L2
                if (i >= 2) {
                    if (!bar_wait(&bars.x_free[b], ph_x[b], &abort_flag, status)) break;
                    ph_x[b] ^= 1;
                }
                mbar_arrive_expect_tx(&bars.x_full[b], kTileBytes);
                tma_load_3d(sb + (b ? L::X1 : L::X0), &tmap_x, 0, t0, bh, &bars.x_full[b]);
            }
        }
    } else if (warp == kWarpMMA || warp == kWarpCons) {
        if (lane == 0) {
            constexpr uint32_t I_PROJ = idesc_bf16(128, L::P, 0, 0);
            constexpr uint32_t I_KV = idesc_bf16(128, 80, 1, 1);
            constexpr uint32_t I_QS = idesc_bf16(128, 80, 0, 0);
            bool ok = true;
            auto wait = [&](uint64_t* bar, uint32_t parity) {
                if (ok) ok = bar_wait(bar, parity, &abort_flag, status);
            };
            auto adv = [](uint64_t d, uint32_t bytes) { return d + (bytes >> 4); };
            const uint64_t d_x[2] = {sdesc(sb + L::X0, 16, 1024), sdesc(sb + L::X1, 16, 1024)};
            const uint64_t d_w = sdesc(sb + L::W, 16, 1024);
            const uint64_t d_pb[2] = {sdesc(sb + L::PB0, 16, 1024), sdesc(sb + L::PB1, 16, 1024)};
            const uint64_t d_pb_mn[2] = {sdesc(sb + L::PB0, 16384, 1024),
                                         sdesc(sb + L::PB1, 16384, 1024)};
            const uint64_t d_v[2] = {sdesc(sb + L::V0, L::VONE - L::V0, 1024),
                                     sdesc(sb + L::V1, L::VONE - L::V1, 1024)};
            const uint64_t d_sx = sdesc(sb + L::SX, 16, 1024);

            auto consume = [&](int j) {  // tensor-core use of the features of job j
                const int i = j / G, g = j % G, fb = j & 1, ib = i & 1;
                wait(&bars.phi_full[fb], (j >> 1) & 1);
                if (MODE == kState) {
                    if (g == 0) wait(&bars.v_full[ib], (i >> 1) & 1);
                    if (!ok) return;
                    fence_after_sync();
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)  // K = 128 tokens
                        mma_bf16(tm + L::T_S + 80 * g, adv(d_pb_mn[fb], ks * 2048),
                                 adv(d_v[ib], ks * 2048), I_KV, (i > 0 || ks > 0) ? 1u : 0u);
                    mma_commit(&bars.phi_free[fb]);
                    if (g == G - 1) mma_commit(&bars.v_free[ib]);
                } else {
                    if (g == 0 && i >= 2) wait(&bars.o_free[ib], ((i - 2) >> 1) & 1);
                    if (!ok) return;
                    fence_after_sync();
                    const uint32_t to = ib ? L::T_O1 : L::T_O0;
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks) {  // K = 128 features of group g
                        const uint32_t kofs = (ks >> 2) * 16384 + (ks & 3) * 32;
                        mma_bf16(tm + to, adv(d_pb[fb], kofs),
                                 adv(d_sx, g * L::SX_GROUP + (ks >> 2) * L::SX_BLOCK + (ks & 3) * 32),
                                 I_QS, (g > 0 || ks > 0) ? 1u : 0u);
                    }
                    mma_commit(&bars.phi_free[fb]);
                    if (g == G - 1) mma_commit(&bars.o_full[ib]);
                }
            };
            // Projections and the state / output MMAs come from two threads, so a late v
            // tile (the state MMA of job j waits for it) never holds up the projection of
            // job j + 2 that the feature warps will want next.
            for (int j = 0; j < njobs && ok && warp == kWarpMMA; ++j) {
                const int i = j / G, g = j % G, pb = j & 1, ib = i & 1;
                if (g == 0) wait(&bars.x_full[ib], (i >> 1) & 1);
                if (j >= 2) wait(&bars.p_free[pb], ((j - 2) >> 1) & 1);
                if (!ok) break;
                fence_after_sync();
                const uint64_t wd = adv(d_w, g * L::P * 128);
#pragma unroll
                for (int ks = 0; ks < 4; ++ks)
                    mma_bf16(tm + (pb ? L::T_P1 : L::T_P0), adv(d_x[ib], ks * 32), adv(wd, ks * 32),
                             I_PROJ, ks > 0);
                mma_commit(&bars.p_full[pb]);
                if (g == G - 1) mma_commit(&bars.x_free[ib]);
            }
            if (warp == kWarpCons) {
                for (int j = 0; j < njobs && ok; ++j) consume(j);
                if (ok && MODE == kState) mma_commit(&bars.state_done);
            }
        }
    } else if (warp < kWarpEW) {
        // ================= features =================
        // Four warps per lane quadrant, each on 16 frequencies of the job's group: with four
        // warps per scheduler one warp's tensor-memory read or sin/cos latency is covered by
        // the others.  Frequencies 16 fq + 2e, + 1 -> pair e of 16-byte chunks 2 fq, 2 fq + 1
        // of the cos and sin blocks.  n: cos(w) by the FMA-pipe polynomial when every argument
        // of the warp is inside [-2, 2].
        const int fq = (warp - kWarpFW) >> 2, quad = warp & 3, t = 32 * quad + lane;
        const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);
        for (int j = 0; j < njobs; ++j) {
            const int i = j / G, pb = j & 1;
            const bool valid = t < min(kC, N - (c0 + i) * kC);
            // state mode: key weight of the norm prefactor (phi(k) scaled by it)
            const float wk = (MODE == kState && KW && valid)
                                 ? kw[(size_t)bh * N + (size_t)(c0 + i) * kC + t] : 1.f;
            if (!bar_wait(&bars.p_full[pb], (j >> 1) & 1, &abort_flag, status)) break;
            fence_after_sync();
            const uint32_t tp = tm_row + (pb ? L::T_P1 : L::T_P0) + 16 * fq;
            float a[16], w[16], ma, mw = 0.f;  // max |x| of each load
            tmem_ld16_maxabs(tp, a, ma);
            if (NS) tmem_ld16_maxabs(tp + 64, w, mw);
            tmem_wait_ld();
            fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars.p_free[pb]);
            if (NS)
                cos_w_args(a, w, fmaxf(ma, mw));  // w <- cos(w)
            else
                reduce_2pi_if_needed(a, ma);
            uint32_t pc[8], ps[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                float s0, cc0, s1, cc1;
                __sincosf(a[2 * e], &s0, &cc0);
                __sincosf(a[2 * e + 1], &s1, &cc1);
                if (NS) {
                    const float cw0 = w[2 * e], cw1 = w[2 * e + 1];
                    cc0 *= cw0; s0 *= cw0; cc1 *= cw1; s1 *= cw1;
                }
                if (MODE == kState && KW) { cc0 *= wk; s0 *= wk; cc1 *= wk; s1 *= wk; }
                if (!valid) { cc0 = s0 = cc1 = s1 = 0.f; }
                pc[e] = pack_bf16(cc0, cc1);
                ps[e] = pack_bf16(s0, s1);
            }
            if (j >= 2 && !bar_wait(&bars.phi_free[pb], ((j - 2) >> 1) & 1, &abort_flag, status))
                break;
            const uint32_t dst = sb + (pb ? L::PB1 : L::PB0);
#pragma unroll
            for (int q = 0; q < 2; ++q) {
                const uint32_t off = swz128(t, (2 * fq + q) * 8);
                st_shared_v4(dst + off, pc[4 * q], pc[4 * q + 1], pc[4 * q + 2], pc[4 * q + 3]);
                st_shared_v4(dst + 16384 + off, ps[4 * q], ps[4 * q + 1], ps[4 * q + 2],
                             ps[4 * q + 3]);
            }
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bars.phi_full[pb]);
        }
    } else {
        // ================= epilogue =================
        const int quad = warp & 3, t = 32 * quad + lane;
        const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);
        if (MODE == kState) {
            if (warp == kWarpEW + 3) {
                // v tiles (tmap_v), issued by this warp's lane 0 before it joins the epilogue
                if (lane == 0) {
                    uint32_t ph_v[2] = {0, 0};
                    for (int i = 0; i < nc; ++i) {
                        const int b = i & 1, t0 = (c0 + i) * kC;
                        if (i + kAhead < nc) tma_prefetch_3d(&tmap_v, 0, t0 + kAhead * kC, bh);
                        if (i >= 2) {
                            if (!bar_wait(&bars.v_free[b], ph_v[b], &abort_flag, status)) break;
                            ph_v[b] ^= 1;
                        }
                        mbar_arrive_expect_tx(&bars.v_full[b], kTileBytes);
                        tma_load_3d(sb + (b ? L::V1 : L::V0), &tmap_v, 0, t0, bh, &bars.v_full[b]);
                    }
                }
                __syncwarp();
            }
            if (bar_wait(&bars.state_done, 0, &abort_flag, status)) {
                fence_after_sync();
                float* dst = part + ((size_t)blockIdx.x * G * 128 + t) * kRow;
                for (int g = 0; g < G; ++g) {
                    float4* d4 = reinterpret_cast<float4*>(dst + (size_t)g * 128 * kRow);
#pragma unroll
                    for (int j = 0; j < 5; ++j) {  // 16 columns at a time (register budget)
                        float s_[16];
                        tmem_ld16(tm_row + L::T_S + 80 * g + 16 * j, s_);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            d4[4 * j + e] = make_float4(s_[4 * e], s_[4 * e + 1], s_[4 * e + 2],
                                                        s_[4 * e + 3]);
                    }
                }
            }
        } else {
            // Output rows are staged as bf16 (128-byte swizzle) in the v tiles, unused in this
            // mode, and written by one TMA store per chunk (tmap_v maps out here): a row per
            // thread straight to global memory puts 32 cache lines in every warp store, and
            // the queue they wait in also holds the feature warps' shared-memory stores.
            // Named barrier 1 joins the 4 epilogue warps; its AND keeps their control flow
            // the same when a wait gives up.
            const bool issuer = warp == kWarpEW && lane == 0;
            for (int i = 0; i < nc; ++i) {
                const int ib = i & 1, t0 = (c0 + i) * kC;
                const bool got = bar_wait(&bars.o_full[ib], (i >> 1) & 1, &abort_flag, status);
                // (the issuer reaches this barrier only after the store that last read
                // staging buffer ib, two chunks back, has read it)
                __syncwarp();
                if (!bar_and(1, 128, got)) break;
                fence_after_sync();
                const uint32_t to = tm_row + (ib ? L::T_O1 : L::T_O0);
                const uint32_t stg = sb + (ib ? L::V1 : L::V0);
                float dn = 0.f, inv = 0.f;
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {  // 32 output columns at a time
                    float o[32];
                    tmem_ld16(to + 32 * hh, *reinterpret_cast<float(*)[16]>(&o[0]));
                    tmem_ld16(to + 32 * hh + 16, *reinterpret_cast<float(*)[16]>(&o[16]));
                    if (hh == 0) dn = tmem_ld1(to + 64);
                    tmem_wait_ld();
                    if (hh == 1) {
                        fence_before_sync();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&bars.o_free[ib]);
                    } else {
                        inv = 1.f / dn;
                    }
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc)
                        st_shared_v4(stg + swz128(t, (4 * hh + cc) * 8),
                                     pack_bf16(o[8 * cc] * inv, o[8 * cc + 1] * inv),
                                     pack_bf16(o[8 * cc + 2] * inv, o[8 * cc + 3] * inv),
                                     pack_bf16(o[8 * cc + 4] * inv, o[8 * cc + 5] * inv),
                                     pack_bf16(o[8 * cc + 6] * inv, o[8 * cc + 7] * inv));
                }
                if (den && t < min(kC, N - t0)) den[(size_t)bh * N + t0 + t] = dn / (float)M;
                fence_proxy_async();
                __syncwarp();
                bar_named(1, 128);
                if (issuer) {
                    tma_store_3d(&tmap_v, stg, 0, t0, bh);  // rows past N are not written
                    bulk_commit_group();
                    bulk_wait_group_read<1>();
                }
            }
            if (issuer) bulk_wait_group<0>();
        }
    }

    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == kWarpMMA) tmem_dealloc(tm, 512);
}

// total[bh][g][f][e] = sum over splits, in split order.
__global__ void nc_reduce_kernel(int BH, int splits, int G, const float* __restrict__ part,
                                 float* __restrict__ total)
{
    const size_t per = (size_t)G * 128 * kRow;
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < (size_t)BH * per;
         idx += (size_t)gridDim.x * blockDim.x) {
        const size_t b = idx / per, e = idx % per;
        const float* p = part + b * splits * per + e;
        float acc = 0.f;
        for (int s = 0; s < splits; ++s) acc += p[(size_t)s * per];
        total[idx] = acc;
    }
}

template <bool NS, int G>
cudaError_t launch_nc(const Problem& p, const void* q, const void* k, const void* v,
                      const float* W1, const float* W2, const float* kw, void* out, float* den,
                      void* scratch, int* status, cudaStream_t s)
{
    const int BH = p.B * p.H, splits = tc_nc_splits(p);
    CUtensorMap mq, mk, mv, mo;
    if (!make_act_map(&mq, q, BH, p.N) || !make_act_map(&mk, k, BH, p.N) ||
        !make_act_map(&mv, v, BH, p.N) || !make_act_map(&mo, out, BH, p.N))
        return cudaErrorInvalidValue;
    float* part = static_cast<float*>(scratch);
    float* total = part + (size_t)BH * splits * G * 128 * kRow;
    const int smem = (int)NcCfg<NS, G>::BYTES + 1024;
    auto k_state = kw ? tc_nc_kernel<kState, NS, G, true> : tc_nc_kernel<kState, NS, G, false>;
    auto k_out = tc_nc_kernel<kOut, NS, G, false>;
    cudaError_t e = cudaFuncSetAttribute(k_state, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_out, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    k_state<<<BH * splits, kThreadsNC, smem, s>>>(mk, mv, p.H, p.N, p.M, splits, W1, W2, kw,
                                                 part, nullptr, nullptr, nullptr, status);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const size_t n = (size_t)BH * G * 128 * kRow;
    nc_reduce_kernel<<<(int)std::min<size_t>((n + 255) / 256, 152 * 8), 256, 0, s>>>(BH, splits, G,
                                                                                    part, total);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    k_out<<<BH * splits, kThreadsNC, smem, s>>>(mq, mo, p.H, p.N, p.M, splits, W1, W2, nullptr,
                                               nullptr, total, (__nv_bfloat16*)out, den, status);
    return cudaGetLastError();
}

}  // namespace

bool tc_nc_supported(const Problem& p)
{
    return p.bf16 && p.d == 64 && (p.M == 64 || p.M == 128) && !p.causal;
}

// Splits per sequence.  A unit costs a fixed set-up (frequencies, tensor memory, pipeline
// fill, partial-state write: about kSetupChunks chunk times, fitted to measured times over
// N = 1K..64K) plus its chunks, and one unit runs per SM at a time; the split count
// minimises waves x (set-up + chunks per unit), at most kTargetUnits units (which bounds
// the partial-state workspace), fewest splits on ties.
int tc_nc_splits(const Problem& p)
{
    const long long BH = (long long)p.B * p.H;
    const int nch = (p.N + kC - 1) / kC;
    const long long smax = std::max(1LL, std::min<long long>(nch, (kTargetUnits + BH - 1) / BH));
    long long best = 1, best_cost = -1;
    for (long long s = 1; s <= smax; ++s) {
        const long long waves = (BH * s + kSMs - 1) / kSMs;
        const long long cost = waves * (kSetupChunks + (nch + s - 1) / s);
        if (best_cost < 0 || cost < best_cost) {
            best_cost = cost;
            best = s;
        }
    }
    return (int)best;
}

size_t tc_nc_ws_bytes(const Problem& p)
{
    const size_t G = (size_t)p.M / 64, BH = (size_t)p.B * p.H;
    return (BH * tc_nc_splits(p) + BH) * G * 128 * kRow * sizeof(float);
}

cudaError_t launch_tc_nc(const Problem& p, const void* q, const void* k, const void* v,
                         const float* W1, const float* W2, const float* kw, void* out,
                         float* den, void* scratch, int* status, cudaStream_t s)
{
    const int G = p.M / 64;
    if (p.nonstat)
        return G == 1 ? launch_nc<true, 1>(p, q, k, v, W1, W2, kw, out, den, scratch, status, s)
                      : launch_nc<true, 2>(p, q, k, v, W1, W2, kw, out, den, scratch, status, s);
    return G == 1 ? launch_nc<false, 1>(p, q, k, v, W1, W2, kw, out, den, scratch, status, s)
                  : launch_nc<false, 2>(p, q, k, v, W1, W2, kw, out, den, scratch, status, s);
}

}  // namespace flex
