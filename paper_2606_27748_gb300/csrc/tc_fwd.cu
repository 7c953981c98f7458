// Causal forward of RFF linear attention on the 5th-generation tensor cores (tcgen05).
//
// Chunked scan of Eq. (linear att) with j <= i: the sequence is cut into chunks of 128
// tokens; inside a chunk the masked kernel matrix A = phi(Q) phi(K)^T is applied directly
// (A V), across chunks the running state S = sum phi(k) v^T and z = sum phi(k) carries the
// prefix (phi(Q) S, phi(Q) z).  phi never leaves the SM: the projection x W^T lands in
// tensor memory, the CUDA cores turn it into cos/sin features (Eq. phi_n, or the product
// form of Eq. phi_non) and hand them to the tensor core: phi(Q) through tensor memory (the
// A operand of phi(Q) phi(K)^T and phi(Q) [S | z]), phi(K) through shared memory.
//
// Frequency groups: each CTA owns one group of 64 frequencies (128 features: 64 cos, then
// 64 sin).  With M = 128 the two groups of a sequence run on the two CTAs of a cluster;
// every term of the numerator and the denominator is a sum over features, so each CTA
// computes a partial [numerator | denominator] over its own features and the pair adds
// the partials through distributed shared memory (CTA r finishes rows 64r..64r+63 of each
// chunk).  Neither CTA ever recomputes the other's features.  Features are unscaled
// ([cos, sin] instead of M^{-1/2}[cos, sin]): the factor cancels in the output, and only
// the stored denominator is rescaled (den = den' / M).
//
// Warp roles, handshakes on mbarriers (896 threads with FW = 16 feature warps; the
// stationary kernel with one CTA per sequence: 640 threads, FW = 8):
//   warp 0      TMA: q and k chunk tiles (128B swizzle) into shared memory
//   warp 1      one thread issues the attention MMAs (numerator, QK, state, A V); owns the
//               tensor-memory allocation
//   warps 2 ..  features: projection (TMEM) -> cos/sin -> phi(Q) into TMEM (bf16 pairs),
//   1 + FW      phi(K) into shared memory; FW / 4 warps per lane quadrant (warp 2 + 4 fq +
//               r'), warp fq on 64 / (FW / 4) frequencies of the group per feature tile (n,
//               per half group of 32: 8 fq .. 8 fq + 7 of the half); with four warps per
//               scheduler the sin/cos unit stays busy while a warp waits on its loads
//   next 8      epilogue, two halves of 4 warps: causal mask + bf16 of A (written back
//               into TMEM as the A operand of A V), bf16 snapshot of [S | z] for the next
//               chunk, partial output rows (own rows, or the partner's rows staged for it)
//   next        one thread issues the projection MMAs, so they never queue behind an
//               attention step that has not been issued yet
//   last        TMA: v chunk tiles (a buffer frees late, after A V, and must not hold up
//               the q and k loads)
//
// Per chunk c the attention issuer runs phi(Q) [S | z] as soon as phi(Q) and the snapshot
// of the state before c are ready, then phi(Q) phi(K)^T and the state update once phi(K)
// is ready, then A V once the epilogue has masked A.  The output accumulator is double
// buffered, so reading out chunk c (and the exchange with the partner) never holds up
// chunk c + 1; the snapshot is taken as soon as the state update of c completes.  The
// nonstationary projection is issued per half group (32 frequencies: 32 u and 32 w
// columns); all feature warps read each half, so the second half is projected while they
// turn the first into features.
//
// Sequence split: when there are SMs to spare, a sequence is cut into `splits` segments
// handled by different CTAs (clusters) with no waiting between them: the CTA of segment j
// first runs a k-only pass over the chunks before its segment (projection + features of k
// and the state update, no outputs) to build the state prefix, then its own chunks.
// Segment lengths halve from one segment to the next, which balances the work because a
// k-only chunk costs about half a full chunk.
//
// z rides in S as an extra column: the state update multiplies phi(K)^T by [V | 1], and
// the output MMAs multiply by [S | z] and [V | 1], so column 64 of the output accumulator
// is the denominator, built from exactly the bf16 values that build the numerator.
//
// Tensor memory (512 columns x 128 lanes, 32-bit):
//   [0,64)     projection (s: a of the 64 frequencies; n: u, w of 32 frequencies, as 4
//              blocks of [u of 8 | w of 8], one per feature warp of a quadrant)
//   [64,192)   A = phi(Q) phi(K)^T (row = query, col = key); after the epilogue, columns
//              [0,32) and [64,96) hold bf16(masked A) of keys 0-63 and 64-127, two per column
//   [192,352)  two buffers of phi(Q) [S | z] + A [V | 1]: numerator 0-63, denominator 64
//   [352,432)  [S | z] (lane = feature), z in column 64
//   [432,496)  phi(Q) as bf16 pairs (column c = features 2c, 2c+1; cos in 0-31, sin 32-63)
#include <cuda.h>

#include "flex_internal.h"
#include "tc_common.cuh"
#include "tc_util.cuh"

namespace flex {
namespace {
using namespace tc;

constexpr int kC = 128;            // tokens per chunk = MMA M
constexpr int kWarpTMA = 0, kWarpMMA = 1, kWarpFW = 2, kEpiWarps = 8;

template <bool NS, int CS>
struct Cfg {
    static constexpr int NH = NS ? 2 : 1;  // projections per feature tile (64 columns each)
    // Feature warps: 16 (four per lane quadrant, 72 registers a thread), except for the
    // stationary kernel with one CTA per sequence: 8 (two per quadrant, 96 registers).  Its
    // features are cheap enough that the attention and epilogue chain sets the chunk
    // period, and that runs faster with the larger budget (measured: 16 warps 0.105 ms,
    // 8 warps 0.094 ms on s_causal B8 H12 N4096; the pair kernels gain from 16).
    static constexpr int FW = (NS || CS > 1) ? 16 : 8;
    static constexpr int EW = kWarpFW + FW;        // first epilogue warp
    static constexpr int PROJ = EW + kEpiWarps;    // projection MMA issuer
    static constexpr int TMAV = PROJ + 1;          // v tiles
    static constexpr int THREADS = 32 * (TMAV + 1);
    // shared memory offsets (bytes, 1024-aligned); X0/X1 hold q/k tiles.  VONE is the
    // second 64-column block of [V | 1] (column 0 = 1, the rest 0), reached from either V
    // buffer through the descriptor's leading byte offset.
    static constexpr uint32_t X0 = 0, X1 = 16384, V0 = 32768, V1 = 49152, VONE = 65536;
    // frequencies, bf16 K-major, 64 rows per projection: s: W rows 0-63; n: half h = rows
    // [U | V] of frequencies 32h + 8fq .. + 7 for fq = 0..3
    static constexpr uint32_t W = 81920;
    static constexpr uint32_t PK = W + 16384;  // phi(K): cos block, sin block (64 features)
    // [S | z] snapshot, MN-major (row = feature): block 0 holds S[f][0..63], block 1 holds
    // z[f] in column 0 and zeros (the MMA reads columns 0-15 of it: N = 80)
    static constexpr uint32_t SX = PK + 32768;
    // Partial [numerator | denominator] exchange with the partner CTA, one block per
    // epilogue warp: 32 rows x 32 numerator columns (128-byte rows, 16-byte chunks
    // swizzled by row), + 32 denominators for the warps with eh = 0.  STG: two buffers of
    // the blocks this CTA sends, XCH: two buffers of the blocks it receives.
    static constexpr uint32_t XNUM = 32 * 128, XBLK0 = XNUM + 32 * 4, XBUF = 2 * (XBLK0 + XNUM);
    static constexpr uint32_t STG = SX + 32768;
    static constexpr uint32_t XCH = STG + 2 * XBUF;
    static constexpr uint32_t BYTES = XCH + 2 * XBUF;
    // tensor memory columns
    static constexpr uint32_t T_P = 0, T_A = 64, T_O = 192, T_S = 352, T_Q = 432;
    static_assert(T_Q + 64 <= 512, "tensor memory budget");
    static_assert(BYTES + 1024 <= 232448, "shared memory budget");
};

struct Bars {
    uint64_t x_full[2], x_free[2], v_full[2], v_free[2];
    uint64_t p_full, p_free, phiq_full, phik_full, phiq_free, phik_free;
    uint64_t attn_done, s_done, a_ready, sx_ready, o_ready, epi_done[2];
    uint64_t xch_full[2];  // the partner's four block copies have landed in XCH (tx count)
    uint64_t never;        // nothing arrives on it (the diagnostic stall)
};

// First chunk of segment j of `splits` (lengths proportional to 2^-j), rounded.
__device__ __forceinline__ int segment_bound(int nch, int splits, int j)
{
    const long long den = (1LL << splits) - 1;
    const long long num = (long long)nch * ((1LL << splits) - (1LL << (splits - j)));
    return (int)((2 * num + den) / (2 * den));
}

// NS: nonstationary features; CS: CTAs per cluster = frequency groups (M / 64); KW: key
// weights of the norm prefactor given (a compile-time switch: the plain kernel is unchanged).
template <bool NS, int CS, bool KW>
__global__ void __launch_bounds__(Cfg<NS, CS>::THREADS, 1)
    tc_fwd_causal_kernel(const __grid_constant__ CUtensorMap tmap_q,
                         const __grid_constant__ CUtensorMap tmap_k,
                         const __grid_constant__ CUtensorMap tmap_v,
                         const __grid_constant__ CUtensorMap tmap_o, int H, int N, int M,
                         int splits, const float* __restrict__ W1,
                         const float* __restrict__ W2, const float* __restrict__ kw,
                         __nv_bfloat16* __restrict__ out, float* __restrict__ den, int* status)
{
    using L = Cfg<NS, CS>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sb = smem_u32(sm);
    __shared__ Bars bars;
    __shared__ uint32_t tmem_base_sh;
    __shared__ volatile int abort_flag;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int rank = CS > 1 ? (int)cluster_rank() : 0;  // = frequency group
    const int unit = blockIdx.x / CS;
    const int bh = unit / splits, seg = unit % splits, h = bh % H;
    const int nch = (N + kC - 1) / kC;
    const int cb = segment_bound(nch, splits, seg), ce = segment_bound(nch, splits, seg + 1);
    if (cb >= ce) return;  // uniform over the cluster
    const size_t base = (size_t)bh * N * 64;

    // ---- set-up: frequencies of the group (bf16, K-major rows), ones, zero snapshot ----
    for (int idx = tid; idx < 128 * 8; idx += L::THREADS) {
        const int r = idx >> 3, c = idx & 7;
        if (!NS && r >= 64) break;
        // n: row r of half h = r/64 belongs to feature warp fq = (r%64)/16: U (r%16 < 8) or
        // V (r%16 >= 8) of frequency 32 h + 8 fq + r%8, so that warp's u and w are the
        // adjacent projection columns 16 fq .. 16 fq + 15
        const int f = 64 * rank + (NS ? 32 * (r >> 6) + 8 * ((r >> 4) & 3) + (r & 7) : r);
        const float* w1 = W1 + ((size_t)h * M + f) * 64 + c * 8;
        float x[8];
        if (!NS) {
#pragma unroll
            for (int e = 0; e < 8; ++e) x[e] = w1[e];
        } else {
            const float* w2 = W2 + ((size_t)h * M + f) * 64 + c * 8;
            const float sgn = (r & 8) ? -1.f : 1.f;  // U = (W1+W2)/2, V = (W1-W2)/2
#pragma unroll
            for (int e = 0; e < 8; ++e) x[e] = 0.5f * (w1[e] + sgn * w2[e]);
        }
        st_shared_v4(sb + L::W + swz128(r, c * 8), pack_bf16(x[0], x[1]), pack_bf16(x[2], x[3]),
                     pack_bf16(x[4], x[5]), pack_bf16(x[6], x[7]));
    }
    for (int idx = tid; idx < 16384 / 16; idx += L::THREADS)  // [1, 0, ..., 0] rows
        st_shared_v4(sb + L::VONE + idx * 16, 0, 0, 0, 0);
    for (int idx = tid; idx < 32768 / 16; idx += L::THREADS)
        st_shared_v4(sb + L::SX + idx * 16, 0, 0, 0, 0);
    __syncthreads();
    for (int r = tid; r < kC; r += L::THREADS)
        *reinterpret_cast<uint16_t*>(sm + L::VONE + swz128(r, 0)) = 0x3F80u;  // bf16 1.0
    if (tid == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars.x_full[i], 1);
            mbar_init(&bars.x_free[i], 1);
            mbar_init(&bars.v_full[i], 1);
            mbar_init(&bars.v_free[i], 1);
            mbar_init(&bars.epi_done[i], kEpiWarps);
        }
        mbar_init(&bars.p_full, 1);
        mbar_init(&bars.p_free, L::FW);
        mbar_init(&bars.phiq_full, L::FW);
        mbar_init(&bars.phik_full, L::FW);
        mbar_init(&bars.phiq_free, 1);
        mbar_init(&bars.phik_free, 1);
        mbar_init(&bars.attn_done, 1);
        mbar_init(&bars.s_done, 1);
        mbar_init(&bars.a_ready, kEpiWarps);
        mbar_init(&bars.sx_ready, kEpiWarps);
        mbar_init(&bars.o_ready, 1);
        mbar_init(&bars.xch_full[0], 1);
        mbar_init(&bars.xch_full[1], 1);
        mbar_init(&bars.never, 1);
        abort_flag = 0;
        fence_mbar_init();
        diagnostic_stall(&bars.never, &abort_flag, status);  // normally returns at once
        if (CS > 1) {  // the first exchange into each buffer
            mbar_arrive_expect_tx(&bars.xch_full[0], L::XBUF);
            mbar_arrive_expect_tx(&bars.xch_full[1], L::XBUF);
        }
    }
    if (warp == kWarpMMA) {
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

    if (abort_flag) {
        // the diagnostic stall ran out during set-up: nothing is issued
    } else if (warp == L::TMAV) {
        // ================= TMA producer: v =================
        if (lane == 0) {
            uint32_t ph_vfree[2] = {0, 0};
            for (int c = 0; c < ce; ++c) {
                const int vb = c & 1;
                if (c >= 2) {
                    if (!bar_wait(&bars.v_free[vb], ph_vfree[vb], &abort_flag, status)) break;
                    ph_vfree[vb] ^= 1;
                }
                if (c + 2 < ce && rank == 0) tma_prefetch_3d(&tmap_v, 0, (c + 2) * kC, bh);
                mbar_arrive_expect_tx(&bars.v_full[vb], kTileBytes);
                tma_load_3d(sb + (vb ? L::V1 : L::V0), &tmap_v, 0, c * kC, bh, &bars.v_full[vb]);
            }
        }
    } else if (warp == kWarpTMA) {
        // ================= TMA producer: q, k =================
        // Main chunks: q -> X0, k -> X1.  k-only prefix chunks alternate k between X1 and
        // X0, so the next tile loads while the current one is projected.
        if (lane == 0) {
            uint32_t ph_xfree[2] = {0, 0};
            bool used_x[2] = {false, false};
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
                if (c + 1 < ce && rank == 0) {  // next chunk's tiles into L2 (once per pair)
                    if (c + 1 >= cb) tma_prefetch_3d(&tmap_q, 0, t0 + kC, bh);
                    tma_prefetch_3d(&tmap_k, 0, t0 + kC, bh);
                }
                if (c >= cb) {
                    if (!load(0, &tmap_q, t0) || !load(1, &tmap_k, t0)) break;
                } else {
                    if (!load((c & 1) ? 0 : 1, &tmap_k, t0)) break;
                }
            }
        }
    } else if (warp == kWarpMMA || warp == L::PROJ) {
        // ================= MMA issue (one thread per role) =================
        if (lane == 0) {
            constexpr uint32_t I_PROJ = idesc_bf16(128, 64, 0, 0);
            constexpr uint32_t I_QK = idesc_bf16(128, 128, 0, 0);
            constexpr uint32_t I_QS = idesc_bf16(128, 80, 0, 1);
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
            if (warp == L::PROJ) {
                // projections: per chunk q (main chunks) then k, each in NH parts
                const uint64_t d_x[2] = {sdesc(sb + L::X0, 16, 1024), sdesc(sb + L::X1, 16, 1024)};
                const uint64_t d_w = sdesc(sb + L::W, 16, 1024);
                uint32_t ph_xfull[2] = {0, 0}, ph_pfree = 0;
                int nproj = 0;
                for (int c = 0; c < ce && ok; ++c) {
                    const bool main = c >= cb;
                    for (int which = main ? 0 : 1; which < 2 && ok; ++which) {
                        const int buf = which == 0 ? 0 : (main ? 1 : ((c & 1) ? 0 : 1));
                        wait(&bars.x_full[buf], ph_xfull[buf]);
                        for (int hf = 0; hf < L::NH && ok; ++hf) {
                            if (nproj > 0) wait(&bars.p_free, ph_pfree);
                            if (!ok) break;
                            fence_after_sync();
                            const uint64_t wd = adv(d_w, hf * 8192);
#pragma unroll
                            for (int ks = 0; ks < 4; ++ks)
                                mma_bf16(tm + L::T_P, adv(d_x[buf], ks * 32), adv(wd, ks * 32),
                                         I_PROJ, ks > 0);
                            mma_commit(&bars.p_full);
                            ++nproj;
                        }
                        mma_commit(&bars.x_free[buf]);
                    }
                }
            } else {
                const uint64_t d_pk = sdesc(sb + L::PK, 16, 1024);
                const uint64_t d_pk_mn = sdesc(sb + L::PK, 16384, 1024);
                const uint64_t d_sx = sdesc(sb + L::SX, 16384, 1024);
                const uint64_t d_v[2] = {sdesc(sb + L::V0, L::VONE - L::V0, 1024),
                                         sdesc(sb + L::V1, L::VONE - L::V1, 1024)};
                uint32_t ph_vfull[2] = {0, 0}, ph_epi[2] = {0, 0};
                uint32_t ph_phiq = 0, ph_phik = 0, ph_aready = 0, ph_sx = 0;
                for (int c = 0; c < ce && ok; ++c) {
                    const bool main = c >= cb;
                    const int kk = c - cb, ob = kk & 1;
                    const uint32_t t_o = L::T_O + 80 * ob;
                    const uint64_t vd = d_v[c & 1];
                    if (main) {
                        // phi(Q) [S | z] (K = 128 features): phi(Q), the snapshot of the
                        // state before this chunk, and a free output buffer
                        wait(&bars.phiq_full, ph_phiq);
                        wait(&bars.sx_ready, ph_sx);
                        if (kk >= 2) wait(&bars.epi_done[ob], ph_epi[ob]);
                        if (!ok) break;
                        fence_after_sync();
#pragma unroll
                        for (int ks = 0; ks < 8; ++ks)
                            mma_bf16_tmem_a(tm + t_o, tm + L::T_Q + 8 * ks, adv(d_sx, ks * 2048),
                                            I_QS, ks > 0);
                    }
                    wait(&bars.phik_full, ph_phik);
                    if (!ok) break;
                    fence_after_sync();
                    if (main) {
#pragma unroll
                        for (int ks = 0; ks < 8; ++ks)  // A = phi(Q) phi(K)^T, K = 128 features
                            mma_bf16_tmem_a(tm + L::T_A, tm + L::T_Q + 8 * ks,
                                            adv(d_pk, (ks >> 2) * 16384 + (ks & 3) * 32), I_QK,
                                            ks > 0);
                        mma_commit(&bars.phiq_free);  // phi(Q) no longer read
                        mma_commit(&bars.attn_done);
                    }
                    wait(&bars.v_full[c & 1], ph_vfull[c & 1]);
                    if (!ok) break;
                    fence_after_sync();
                    const uint32_t acc_s = c > 0 ? 1u : 0u;
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)  // [S | z] += phi(K)^T [V | 1], K = 128 tokens
                        mma_bf16(tm + L::T_S, adv(d_pk_mn, ks * 2048), adv(vd, ks * 2048), I_KV,
                                 (acc_s | (ks > 0)) ? 1u : 0u);
                    mma_commit(&bars.phik_free);  // phi(K) no longer read
                    if (main || c == cb - 1) mma_commit(&bars.s_done);
                    if (!main) {
                        mma_commit(&bars.v_free[c & 1]);
                        continue;
                    }
                    wait(&bars.a_ready, ph_aready);
                    if (!ok) break;
                    fence_after_sync();
#pragma unroll
                    for (int ks = 0; ks < 8; ++ks)  // keys 16ks..16ks+15: bf16 A columns
                        mma_bf16_tmem_a(tm + t_o, tm + L::T_A + 64 * (ks >> 2) + 8 * (ks & 3),
                                        adv(vd, ks * 2048), I_AV, 1u);
                    mma_commit(&bars.o_ready);
                    mma_commit(&bars.v_free[c & 1]);
                }
            }
        }
    } else if (warp < L::EW) {
        // ================= features =================
        // FW / 4 warps per lane quadrant; warp fq of a quadrant covers FQ = 64 / (FW / 4)
        // frequencies of the group per feature tile.  n (FW = 16): per half r (one projection
        // of 32 frequencies) it reads columns 16 fq .. + 15 = u then w of frequencies
        // 32 r + 8 fq .. + 7; s: the one projection's columns FQ fq .. + FQ - 1 = a of those
        // frequencies.  Each 16-column load returns its max |x| for the range test.
        static_assert(!NS || L::FW == 16, "n: the W rows are ordered for four warps per quadrant");
        constexpr int FQ = 256 / L::FW;  // frequencies per warp per tile (16 or 32)
        constexpr int NL = NS ? 1 : FQ / 16;  // 16-column loads per projection
        constexpr int NPR = NS ? 4 : 8 * NL;  // bf16 pairs per projection
        const int fq = (warp - kWarpFW) >> 2, quad = warp & 3, t = 32 * quad + lane;
        const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);
        uint32_t ph_pfull = 0;
        int n = 0, nq = 0;  // k and q feature tiles produced so far
        for (int c = 0; c < ce; ++c) {
            const bool main = c >= cb;
            const bool valid = t < min(kC, N - c * kC);
            // key weight of the norm prefactor (phi(k) scaled by it), loaded early
            const float wk = (KW && valid) ? kw[(size_t)bh * N + (size_t)c * kC + t] : 1.f;
            for (int which = main ? 0 : 1; which < 2; ++which) {  // 0: q, 1: k
                // bf16 pairs: pair p = frequencies 2p, 2p + 1 of the warp's FQ (n: pairs
                // 4r .. 4r + 3 from half r)
                uint32_t pc[FQ / 2], ps[FQ / 2];
#pragma unroll
                for (int r = 0; r < L::NH; ++r) {
                    if (!bar_wait(&bars.p_full, ph_pfull, &abort_flag, status)) goto fw_out;
                    ph_pfull ^= 1;
                    fence_after_sync();
                    float x[NL][16], mabs[NL];
#pragma unroll
                    for (int l = 0; l < NL; ++l)
                        tmem_ld16_maxabs(tm_row + L::T_P + 16 * (NL * fq + l), x[l], mabs[l]);
                    tmem_wait_ld();
                    fence_before_sync();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&bars.p_free);
#pragma unroll
                    for (int l = 0; l < NL; ++l) {
                        if (NS)  // x[l][8 ..] <- cos(w)
                            cos_w_args(*reinterpret_cast<float(*)[8]>(&x[l][0]),
                                       *reinterpret_cast<float(*)[8]>(&x[l][8]), mabs[l]);
                        else
                            reduce_2pi_if_needed(x[l], mabs[l]);
                    }
#pragma unroll
                    for (int i = 0; i < NPR; ++i) {
                        const float* xl = x[NS ? 0 : i / 8];
                        const int e = NS ? 2 * i : 2 * (i % 8);
                        float s0, c0, s1, c1;
                        __sincosf(xl[e], &s0, &c0);
                        __sincosf(xl[e + 1], &s1, &c1);
                        if (NS) {
                            const float cw0 = xl[8 + e], cw1 = xl[8 + e + 1];
                            c0 *= cw0; s0 *= cw0; c1 *= cw1; s1 *= cw1;
                        }
                        if (KW && which == 1) { c0 *= wk; s0 *= wk; c1 *= wk; s1 *= wk; }
                        if (!valid) { c0 = s0 = c1 = s1 = 0.f; }
                        pc[NPR * r + i] = pack_bf16(c0, c1);
                        ps[NPR * r + i] = pack_bf16(s0, s1);
                    }
                }
                if (which == 0) {
                    // phi(Q) -> tensor memory once the previous chunk's MMAs that read it
                    // are done; column = frequency / 2 (cos), 32 + frequency / 2 (sin)
                    if (nq > 0 && !bar_wait(&bars.phiq_free, (nq - 1) & 1, &abort_flag, status))
                        goto fw_out;
                    fence_after_sync();
                    if (NS) {
#pragma unroll
                        for (int r = 0; r < 2; ++r) {
                            tmem_st4(tm_row + L::T_Q + 16 * r + 4 * fq, &pc[4 * r]);
                            tmem_st4(tm_row + L::T_Q + 32 + 16 * r + 4 * fq, &ps[4 * r]);
                        }
                    } else {
#pragma unroll
                        for (int l = 0; l < NL; ++l) {
                            tmem_st8(tm_row + L::T_Q + FQ / 2 * fq + 8 * l, &pc[8 * l]);
                            tmem_st8(tm_row + L::T_Q + 32 + FQ / 2 * fq + 8 * l, &ps[8 * l]);
                        }
                    }
                    tmem_wait_st();
                    fence_before_sync();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&bars.phiq_full);
                    ++nq;
                } else {
                    if (n > 0 && !bar_wait(&bars.phik_free, (n - 1) & 1, &abort_flag, status))
                        goto fw_out;
                    // 16-byte chunk m = frequencies 8 m .. 8 m + 7: n: m = 4 j + fq (j = half),
                    // s: m = FQ / 8 fq + j
#pragma unroll
                    for (int j = 0; j < FQ / 8; ++j) {
                        const uint32_t off = swz128(t, (NS ? 4 * j + fq : FQ / 8 * fq + j) * 8);
                        st_shared_v4(sb + L::PK + off, pc[4 * j], pc[4 * j + 1], pc[4 * j + 2],
                                     pc[4 * j + 3]);
                        st_shared_v4(sb + L::PK + 16384 + off, ps[4 * j], ps[4 * j + 1],
                                     ps[4 * j + 2], ps[4 * j + 3]);
                    }
                    fence_proxy_async();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&bars.phik_full);
                    ++n;
                }
            }
        }
    fw_out:;
    } else {
        // ================= epilogue =================
        // Two halves of 4 warps (one warp per lane quadrant each): half eh takes keys
        // [64eh, 64eh+64) of A, output columns [32eh, 32eh+32) and state columns
        // [32eh, 32eh+32) (+ z for eh = 0).  With a partner CTA, a warp on the partner's
        // rows stages its partial block and bulk-copies it into the partner's XCH; a warp on
        // the own rows adds the partner's block once it has landed.
        const int eh = (warp - L::EW) >> 2, quad = warp & 3, t = 32 * quad + lane;
        const uint32_t tm_row = tm + ((uint32_t)(32 * quad) << 16);
        const int partner = rank ^ 1;
        const bool own_rows = CS == 1 || (quad >> 1) == rank;
        const uint32_t xblk = (quad & 1) * (L::XBLK0 + L::XNUM) + eh * L::XBLK0;  // this warp's
        const uint32_t xrow = xblk + 128 * lane;                                  // block
        uint32_t ph_attn = 0, ph_s = 0, ph_o = 0, ph_xfull[2] = {0, 0};
        auto signal = [&](uint64_t* bar) {
            fence_proxy_async();
            fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar);
        };
        auto snapshot = [&]() -> bool {
            // MN-major [S | z]: row f (= this thread's lane = feature) holds S[f][.]
            if (!bar_wait(&bars.s_done, ph_s, &abort_flag, status)) return false;
            ph_s ^= 1;
            fence_after_sync();
            float s_[32];
            tmem_ld16(tm_row + L::T_S + 32 * eh, *reinterpret_cast<float(*)[16]>(&s_[0]));
            tmem_ld16(tm_row + L::T_S + 32 * eh + 16, *reinterpret_cast<float(*)[16]>(&s_[16]));
            const float zz = eh == 0 ? tmem_ld1(tm_row + L::T_S + 64) : 0.f;
            tmem_wait_ld();
#pragma unroll
            for (int v = 0; v < 4; ++v)
                st_shared_v4(sb + L::SX + swz128(t, 32 * eh + 8 * v),
                             pack_bf16(s_[8 * v], s_[8 * v + 1]), pack_bf16(s_[8 * v + 2], s_[8 * v + 3]),
                             pack_bf16(s_[8 * v + 4], s_[8 * v + 5]),
                             pack_bf16(s_[8 * v + 6], s_[8 * v + 7]));
            if (eh == 0) st_shared_v4(sb + L::SX + 16384 + swz128(t, 0), pack_bf16(zz, 0.f), 0, 0, 0);
            signal(&bars.sx_ready);
            return true;
        };
        if (cb > 0) {  // the k-only prefix ends here: snapshot its state
            if (!snapshot()) goto ew_out;
        } else {
            signal(&bars.sx_ready);  // zero state
        }
        for (int c = cb; c < ce; ++c) {
            const int t0 = c * kC, kk = c - cb;
            const bool valid = t < min(kC, N - t0);
            if (!bar_wait(&bars.attn_done, ph_attn, &abort_flag, status)) goto ew_out;
            ph_attn ^= 1;
            fence_after_sync();
            // Causal mask + bf16 of the two 32-key blocks kb = 2 eh + b of this half: a block
            // above the diagonal block of this warp's rows (kb > quad) is zeros (nothing
            // loaded), the diagonal block (kb = quad) keeps j <= i, a block below it
            // (kb < quad) is copied.  Block b's bf16 pairs go to columns 64 eh + 16 b .. + 15,
            // which this thread read with block 0.
            if constexpr (L::FW == 16) {
                // one block at a time (72-register budget)
#pragma unroll 1
                for (int b = 0; b < 2; ++b) {
                    const int kb = 2 * eh + b;
                    uint32_t pk[16];
                    if (kb <= quad) {
                        float a[32];
                        tmem_ld16(tm_row + L::T_A + 32 * kb, *reinterpret_cast<float(*)[16]>(&a[0]));
                        tmem_ld16(tm_row + L::T_A + 32 * kb + 16,
                                  *reinterpret_cast<float(*)[16]>(&a[16]));
                        tmem_wait_ld();
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const int j0 = 32 * kb + 2 * i;
                            pk[i] = kb < quad ? pack_bf16(a[2 * i], a[2 * i + 1])
                                              : pack_bf16(j0 <= t ? a[2 * i] : 0.f,
                                                          j0 + 1 <= t ? a[2 * i + 1] : 0.f);
                        }
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) pk[i] = 0u;
                    }
                    tmem_st16(tm_row + L::T_A + 64 * eh + 16 * b, pk);
                }
            } else {
                // block 1 is loaded while block 0 is stored
                auto convert = [&](const float (&a)[32], int kb, uint32_t (&pk2)[16]) {
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int j0 = 32 * kb + 2 * i;
                        pk2[i] = kb < quad ? pack_bf16(a[2 * i], a[2 * i + 1])
                                           : pack_bf16(j0 <= t ? a[2 * i] : 0.f,
                                                       j0 + 1 <= t ? a[2 * i + 1] : 0.f);
                    }
                };
                const int kb0 = 2 * eh, kb1 = kb0 + 1;
                uint32_t pk0[16], pk1[16];
                float a[32];
                if (kb0 <= quad) {
                    tmem_ld16(tm_row + L::T_A + 32 * kb0, *reinterpret_cast<float(*)[16]>(&a[0]));
                    tmem_ld16(tm_row + L::T_A + 32 * kb0 + 16,
                              *reinterpret_cast<float(*)[16]>(&a[16]));
                    tmem_wait_ld();
                    convert(a, kb0, pk0);
                } else {
#pragma unroll
                    for (int i = 0; i < 16; ++i) pk0[i] = 0u;
                }
                if (kb1 <= quad) {  // load block 1 before storing block 0 over its columns'
                                    // neighbours (the store targets columns already read)
                    tmem_ld16(tm_row + L::T_A + 32 * kb1, *reinterpret_cast<float(*)[16]>(&a[0]));
                    tmem_ld16(tm_row + L::T_A + 32 * kb1 + 16,
                              *reinterpret_cast<float(*)[16]>(&a[16]));
                }
                tmem_st16(tm_row + L::T_A + 64 * eh, pk0);
                if (kb1 <= quad) {
                    tmem_wait_ld();
                    convert(a, kb1, pk1);
                } else {
#pragma unroll
                    for (int i = 0; i < 16; ++i) pk1[i] = 0u;
                }
                tmem_st16(tm_row + L::T_A + 64 * eh + 16, pk1);
            }
            tmem_wait_st();
            signal(&bars.a_ready);
            if (c + 1 < ce && !snapshot()) goto ew_out;

            if (!bar_wait(&bars.o_ready, ph_o, &abort_flag, status)) goto ew_out;
            ph_o ^= 1;
            fence_after_sync();
            const uint32_t t_o = L::T_O + 80 * (kk & 1);
            float o[32];
            tmem_ld16(tm_row + t_o + 32 * eh, *reinterpret_cast<float(*)[16]>(&o[0]));
            tmem_ld16(tm_row + t_o + 32 * eh + 16, *reinterpret_cast<float(*)[16]>(&o[16]));
            float dn = tmem_ld1(tm_row + t_o + 64);
            tmem_wait_ld();
            const int xb = kk & 1;
            if (!own_rows) {
                // Partials of the partner's rows -> staging block -> partner's XCH[xb].  Both
                // buffers are free without a handshake: the partner read XCH[xb] two chunks
                // ago before it masked the next chunk, which this CTA's A V has waited for
                // through the exchange of the chunk in between; the same chain orders the
                // copy out of this staging buffer two chunks ago before this write.
                const uint32_t stg = sb + L::STG + xb * L::XBUF;
#pragma unroll
                for (int cc = 0; cc < 8; ++cc)
                    st_shared_v4(stg + xrow + ((cc ^ (lane & 7)) << 4), __float_as_uint(o[4 * cc]),
                                 __float_as_uint(o[4 * cc + 1]), __float_as_uint(o[4 * cc + 2]),
                                 __float_as_uint(o[4 * cc + 3]));
                if (eh == 0) *reinterpret_cast<float*>(sm + (stg - sb) + xblk + L::XNUM + 4 * lane) = dn;
                fence_proxy_async();
                __syncwarp();
                if (lane == 0)
                    bulk_copy_cluster(mapa(sb + L::XCH + xb * L::XBUF + xblk, partner), stg + xblk,
                                      eh == 0 ? L::XBLK0 : L::XNUM,
                                      mapa(smem_u32(&bars.xch_full[xb]), partner));
                __syncwarp();
            }
            signal(&bars.epi_done[kk & 1]);  // this output buffer may be reused
            if (own_rows) {
                if (CS > 1) {
                    if (!bar_wait(&bars.xch_full[xb], ph_xfull[xb], &abort_flag, status))
                        goto ew_out;
                    ph_xfull[xb] ^= 1;
                    const uint8_t* blk = sm + L::XCH + xb * L::XBUF + xrow;
#pragma unroll
                    for (int cc = 0; cc < 8; ++cc) {
                        const float4 p4 =
                            *reinterpret_cast<const float4*>(blk + ((cc ^ (lane & 7)) << 4));
                        o[4 * cc] += p4.x;
                        o[4 * cc + 1] += p4.y;
                        o[4 * cc + 2] += p4.z;
                        o[4 * cc + 3] += p4.w;
                    }
                    // the denominator block travels with the eh = 0 warps' blocks
                    dn += *reinterpret_cast<const float*>(sm + L::XCH + xb * L::XBUF +
                                                          (quad & 1) * (L::XBLK0 + L::XNUM) +
                                                          L::XNUM + 4 * lane);
                    // the warp on rows 0-31 of this half arms this buffer's next exchange
                    if (lane == 0 && (quad & 1) == 0 && eh == 0 && c + 2 < ce)
                        mbar_arrive_expect_tx(&bars.xch_full[xb], L::XBUF);
                }
                if constexpr (CS == 1) {
                    // This warp's 32 x 32 block of out goes through its own staging tile in
                    // the (here unused) exchange region and one TMA store: rows written one
                    // per thread straight to global memory put 32 cache lines in each warp
                    // store, and the memory-instruction queue they fill also carries the
                    // issuers' mbarrier waits.  Rows past N are not written by the store.
                    const uint32_t stg = sb + L::STG + ((warp - L::EW) * 2 + xb) * 2048;
                    const float inv = 1.f / dn;
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc)
                        st_shared_v4(stg + swz64(lane, cc),
                                     pack_bf16(o[8 * cc] * inv, o[8 * cc + 1] * inv),
                                     pack_bf16(o[8 * cc + 2] * inv, o[8 * cc + 3] * inv),
                                     pack_bf16(o[8 * cc + 4] * inv, o[8 * cc + 5] * inv),
                                     pack_bf16(o[8 * cc + 6] * inv, o[8 * cc + 7] * inv));
                    if (valid && den && eh == 0) den[(size_t)bh * N + t0 + t] = dn / (float)M;
                    fence_proxy_async();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_3d(&tmap_o, stg, 32 * eh, t0 + 32 * quad, bh);
                        bulk_commit_group();
                        bulk_wait_group_read<1>();  // the other staging tile is free again
                    }
                    __syncwarp();
                } else if (valid) {
                    const float inv = 1.f / dn;
                    uint4* dst =
                        reinterpret_cast<uint4*>(out + base + (size_t)(t0 + t) * 64 + 32 * eh);
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc)
                        dst[cc] = make_uint4(pack_bf16(o[8 * cc] * inv, o[8 * cc + 1] * inv),
                                             pack_bf16(o[8 * cc + 2] * inv, o[8 * cc + 3] * inv),
                                             pack_bf16(o[8 * cc + 4] * inv, o[8 * cc + 5] * inv),
                                             pack_bf16(o[8 * cc + 6] * inv, o[8 * cc + 7] * inv));
                    if (den && eh == 0) den[(size_t)bh * N + t0 + t] = dn / (float)M;
                }
            }
        }
    ew_out:
        if (CS == 1 && lane == 0) bulk_wait_group<0>();  // stores done before the CTA exits
    }

    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    if (warp == kWarpMMA) tmem_dealloc(tm, 512);
    if (CS > 1) cluster_sync();  // no CTA leaves while its partner may still write to it
}

template <bool NS, int CS, bool KW>
cudaError_t launch_one(const Problem& p, const void* q, const void* k, const void* v,
                       const float* W1, const float* W2, const float* kw, void* out,
                       float* den, int* status, cudaStream_t s)
{
    CUtensorMap mq, mk, mv;
    const int BH = p.B * p.H;
    CUtensorMap mo;
    if (!make_act_map(&mq, q, BH, p.N) || !make_act_map(&mk, k, BH, p.N) ||
        !make_act_map(&mv, v, BH, p.N) || !make_out_map32(&mo, out, BH, p.N))
        return cudaErrorInvalidValue;
    const int splits = tc_fwd_splits(p, sm_count());
    auto kern = tc_fwd_causal_kernel<NS, CS, KW>;
    const int smem = (int)Cfg<NS, CS>::BYTES + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(BH * splits * CS));
    cfg.blockDim = dim3(Cfg<NS, CS>::THREADS);
    cfg.dynamicSmemBytes = (size_t)smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, mq, mk, mv, mo, p.H, p.N, p.M, splits, W1, W2, kw,
                              (__nv_bfloat16*)out, den, status);
}

}  // namespace

int tc_fwd_splits(const Problem& p, int sms)
{
    const long long units = (long long)p.B * p.H * (p.M / 64);  // CTAs per segment
    const int nch = (p.N + kC - 1) / kC;
    if (sms > 0 && 3 * units <= sms && nch >= 14) return 3;
    if (sms > 0 && 2 * units <= sms && nch >= 6) return 2;
    return 1;
}

bool tc_fwd_supported(const Problem& p)
{
    return p.bf16 && p.d == 64 && (p.M == 64 || p.M == 128) && p.causal;
}

cudaError_t launch_tc_fwd(const Problem& p, const void* q, const void* k, const void* v,
                          const float* W1, const float* W2, const float* kw, void* out,
                          float* den, int* status, cudaStream_t s)
{
    const bool pair = p.M == 128;
    if (kw) {
        if (p.nonstat)
            return pair ? launch_one<true, 2, true>(p, q, k, v, W1, W2, kw, out, den, status, s)
                        : launch_one<true, 1, true>(p, q, k, v, W1, W2, kw, out, den, status, s);
        return pair ? launch_one<false, 2, true>(p, q, k, v, W1, W2, kw, out, den, status, s)
                    : launch_one<false, 1, true>(p, q, k, v, W1, W2, kw, out, den, status, s);
    }
    if (p.nonstat)
        return pair ? launch_one<true, 2, false>(p, q, k, v, W1, W2, kw, out, den, status, s)
                    : launch_one<true, 1, false>(p, q, k, v, W1, W2, kw, out, den, status, s);
    return pair ? launch_one<false, 2, false>(p, q, k, v, W1, W2, kw, out, den, status, s)
                : launch_one<false, 1, false>(p, q, k, v, W1, W2, kw, out, den, status, s);
}

}  // namespace flex
