// fwd_mma.cu -- forward pass on tensor cores (mma.sync, m16n8) with TMA
// staging (arXiv 2606.28560, Section 2 "Attended set").
//
// A warp owns one 16-row tile of queries, tiles placed every 15 queries (the
// 16th row duplicates the next tile's first query and is discarded), so for a
// rung with floor s0 the 16 slab rows [b-s0-1, b-s0+15) hold both rows every
// valid query of the tile reads: query u reads slab row u (far, weight w) and
// row u+1 (floor, weight 1-w).  Scores:
//   window band  S = Q~ K~[b-Wp, b+16)^T   (16 x (16+Wp), the causal band t=0..W)
//   rung k       S = Q~ K~[b-s0-1, +16)^T (16 x 16; the diagonal and the first
//                superdiagonal are the far and floor scores)
// The interpolated rung score (1-w) S[u][u+1] + w S[u][u] is held by at most
// two lanes of the quad that shares a row (one shuffle between them).  The q~
// fragments carry scale * log2(e), so scores are in log2 units.  Softmax is
// two-pass in registers (row max, then P = 2^(s - max)); the
// probability-weighted values are again 16x8 MMAs:
//   window band  O += P_band V[b-Wp, b+16)
//   rung k       O += Phat_k V[b-s0-1, +16),  Phat_k[u][u] = p w, Phat_k[u][u+1] = p (1-w)
// and one more MMA per k-step against a B fragment of ones gives the row sums.
//
// Precision (bf16 I/O): q~ and k~ enter the score MMAs as fp16 (11-bit
// significands); P of the window band is the unnormalised exp(s - max) in
// bf16, so the largest entry of each row is exactly 1; the entries p w and
// p (1-w) of a rung's Phat are rounded to bf16 the same way.  Row sums add
// the same rounded values, so each output is a normalised average of the
// values.  Accumulation is fp32.
//
// Staging: the CTA's union of key rows (rotated keys, fp16) and then of value
// rows (bf16, same buffer) is copied by TMA (3-D tensor maps [heads][T][64],
// 64-row boxes with 8-row tails, 128-byte swizzle, rows outside [0, T)
// zero-filled) under mbarriers with bounded waits; the value copies are
// issued by the last warp done with the keys.  The one-head form writes its
// output rows (and the rotated query rows it keeps) through a 1 KB stage per
// warp, as 16-byte pieces of runs of consecutive rows.
#include <cmath>

#include <cuda.h>
#include <cudaTypedefs.h>

#include "fibattn_internal.cuh"
#include "fwd_mma.cuh"
#include "mma_common.cuh"

namespace fibattn {
namespace {

using namespace mma;

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kWarps = kMmaWarps;
constexpr int kRowsPerWarp = 15;                 // useful query rows of a 16-row tile

// TEAMS = 1: a CTA of 8 warps computes one query head's tile; keys and then
// values are staged into one buffer.  TEAMS = 2 (grouped-query attention): a
// CTA of 16 warps owns a kv head's tile; keys and values are staged once, into
// two buffers, and each team of 8 warps loops over its share of the group's
// query heads (team t takes heads t, t + 2, ...).
// SAVE: also write the residuals the tensor-core backward reads instead of
// recomputing the scores, each where it is formed -- the rotated queries, the
// unnormalised p = exp(s - max) of every slot (fp32, 0 where not attended),
// the far-minus-floor raw score of every rung and 1 / (row sum) per query.
template <int NT, int TEAMS, bool SAVE>
__global__ void __launch_bounds__(kWarps * 32 * TEAMS, TEAMS == 1 ? 2 : 1)
fwd_mma_kernel(const __grid_constant__ RowMaps tmK, const __grid_constant__ RowMaps tmV,
               FwdArgs a, MmaLayout L) {
    // The kernel before this one is the key rotation of the same call, which
    // writes only the rotated keys: the query rows are loaded before waiting
    // for it (TEAMS = 1; the grouped form waits at once).
    pdl_trigger();
    if (TEAMS == 2) pdl_wait();
    constexpr int Wp = NT * 8 - 16;               // window rows before the tile
    extern __shared__ unsigned char smem_raw[];
    __shared__ unsigned long long bars[2];
    // TEAMS = 1, per warp: 8 output rows on their way out (the grouped form,
    // one 16-warp CTA per SM, stores directly: the stage's shared memory costs
    // it more L1 than the scattered stores do)
    __shared__ __align__(16) unsigned ostage[TEAMS == 1 ? kWarps : 1][256];
    unsigned char* buf = reinterpret_cast<unsigned char*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    unsigned char* vbuf = TEAMS == 1 ? buf : buf + (size_t)L.rows * 128;
    const unsigned sbase = smem_u32(buf), vbase = smem_u32(vbuf);

    const Shape& s = a.s;
    // block = unit * tiles + tile; unit = query head (b H + h), or kv head (b Hkv + hk) for TEAMS = 2
    const int unit = (int)fdiv(blockIdx.x, s.dTiles);
    const int i0 = ((int)blockIdx.x - unit * (int)s.dTiles.d) * kMmaTile;
    const int b = (int)fdiv((unsigned)unit, TEAMS == 1 ? s.dH : s.dHkv);
    const int hk = TEAMS == 1 ? (int)fdiv((unsigned)(unit - b * s.H), s.dG) : unit - b * s.Hkv;
    const int head = b * s.Hkv + hk;
    const int tid = threadIdx.x, lane = tid & 31, warp = (tid >> 5) % kWarps, team = (tid >> 5) / kWarps;
    const int g4 = lane >> 2, c4 = lane & 3;
    const int wrel = warp * kRowsPerWarp;         // tile-relative first row of this warp
    const int bw = i0 + wrel;                     // absolute first row

    // raw q words of this thread (rows g4, g4+8; dims 16kc + 2c4.. and 16kc + 8 + 2c4..)
    unsigned qraw[2][4][2];
    auto load_q = [&](int bhq) {
        const __nv_bfloat16* Q = reinterpret_cast<const __nv_bfloat16*>(a.q) + ((size_t)bhq * s.T) * kHeadDim;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const __nv_bfloat16* row = Q + (size_t)min(bw + g4 + 8 * half, s.T - 1) * kHeadDim;
#pragma unroll
            for (int kc = 0; kc < 4; ++kc) {
                qraw[half][kc][0] = *reinterpret_cast<const unsigned*>(row + 16 * kc + 2 * c4);
                qraw[half][kc][1] = *reinterpret_cast<const unsigned*>(row + 16 * kc + 8 + 2 * c4);
            }
        }
    };
    if (TEAMS == 1) {
        load_q(unit);
        pdl_wait();
    }

    // ---- issue the key copies (and for TEAMS = 2 the value copies) (warp 0,
    // once the barriers are initialised; the other warps go on to their q~)
    __shared__ unsigned keys_done;                // warps done with the staged keys (TEAMS = 1)
    __shared__ RopeSmem rsm;
    rope_to_smem(rsm, a.rope, L, tid);
    if (tid == 0) {
        mbar_init(&bars[0], 1);
        mbar_init(&bars[1], 1);
        keys_done = 0;
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    __syncthreads();                              // barrier init visible
    if (tid < 32) {
        issue_rows(buf, &tmK.m64, &tmK.m8, L, i0, head, &bars[0], lane);
        if (TEAMS == 2) issue_rows(vbuf, &tmV.m64, &tmV.m8, L, i0, head, &bars[1], lane);
    }
    // A warp whose tile starts past the end of the sequence (the last tile of
    // a head) has no query to compute; in the one-head form it still counts
    // as done with the keys, and issues the value copies if it is the last.
    if (bw >= s.T) {
        if (TEAMS == 1) {
            __syncwarp();
            unsigned before = 0;
            if (lane == 0) before = atom_add_acq_rel(&keys_done, 1u);
            before = __shfl_sync(0xffffffffu, before, 0);
            if (before == kWarps - 1) {
                asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
                issue_rows(buf, &tmV.m64, &tmV.m8, L, i0, head, &bars[1], lane);
            }
        }
        return;
    }

    // ---- per-lane constants of the fragment layouts
    // ldmatrix (keys, non-transposed): lane supplies row lr of matrix lh; the
    // swizzled chunk of a row r is chunk ^ (r & 7), so for the 8-row groups of
    // one load the address is base(r) with (lh ^ r) & 7, and the loads of the
    // next 8 rows (+1024 bytes) and of chunks 4..7 (address bit 6) follow.
    const int lr = lane & 7, lh = lane >> 3;
    // ldmatrix .trans (values): lane supplies row lv of the 16-row k-chunk and
    // chunk n + lq of it (n even, so chunk n + lq = n ^ lq).
    const int lv = (lane & 7) + (lane & 8), lq = lane >> 4;
    // Rung columns: slab rows x = 0..15 at absolute bw - s0 - 1 + x.  Row r's
    // far score is column x = r (weight w), its floor score column x = r + 1
    // (weight 1-w).  Of this thread's entries (rows g4, g4+8; columns 2c4,
    // 2c4+1 and 2c4+8, 2c4+9) only those with x - r in {-1, 0, 1} can be
    // either, a pattern fixed by delta = 2c4 - g4: entries (g4, 2c4 + u) and
    // (g4+8, 2c4+8 + u) take  u=0: w if delta = 0, 1-w if delta = 1;
    //                         u=1: w if delta = -1, 1-w if delta = 0,
    // each of the form A + B w; row g4 = 7 also has its floor at column 8.
    // The same weights place p in the A fragment of the value product, and B
    // alone (the derivative in w) gives the far-minus-floor score.
    const int dl = 2 * c4 - g4;
    const float ia0 = dl == 1 ? 1.f : 0.f, ib0 = dl == 0 ? 1.f : (dl == 1 ? -1.f : 0.f);
    const float ia1 = dl == 0 ? 1.f : 0.f, ib1 = dl == -1 ? 1.f : (dl == 0 ? -1.f : 0.f);
    const float m7 = (g4 == 7 && c4 == 0) ? 1.f : 0.f;
    // A row's rung score lives in at most two lanes of its quad: for even g4
    // lane g4/2 holds both columns; for odd g4 lanes (g4-1)/2 and (g4+1)/2
    // (lanes 3 and 0 for g4 = 7) hold one each.  One shuffle from the partner
    // lane completes the sum in both; a lane with no column of the row adds a
    // partial of zero and takes no part in the softmax of that row.
    const bool contrib = (dl >= -1 && dl <= 1) || m7 != 0.f;
    const bool writer = dl == 0 || dl == -1;      // one lane per row stores its residuals
    int partner;
    if (g4 & 1) {
        const int x = (g4 - 1) >> 1, y = ((g4 + 1) >> 1) & 3;
        partner = c4 == x ? y : (c4 == y ? x : c4);
    } else {
        partner = ((g4 >> 1) + 1) & 3;
    }
    const int src = (lane & ~3) | partner;

#pragma unroll 1
    for (int hq = TEAMS == 1 ? 0 : team; hq < (TEAMS == 1 ? 1 : s.G); hq += TEAMS) {
    const int bh = TEAMS == 1 ? unit : b * s.H + hk * s.G + hq;

    // ---- q~ as fp16 A fragments (rows g4, g4+8 of the tile; RoPE pairs m, m+32),
    // pre-scaled by scale * log2(e) so that the scores come out in log2 units.
    // Thread dims: 16kc + 2c4 + {0,1} and 16kc + 8 + 2c4 + {0,1} for kc = 0..3.
    // SAVE: also q~ itself as bf16 (qs), the residual the key pass reads.
    const float sc2 = s.scale * kLog2e;
    unsigned qa[4][4], qs[SAVE ? 4 : 1][4];
    float qmax = 0.f;                             // largest |fp16 operand| of the thread: fp16 holds < 65520
    {
        if (TEAMS == 2) load_q(bh);
        // cos/sin of the 8 pairs at position bw+g4, then advanced by 8 positions
        // for row g4+8 with the host's fp64 cos/sin(8 theta_m); they carry the
        // score scale (the SAVE residual divides it out again)
        float cs[2][4], sn[2][4];
        const int pos0 = bw + g4;
        const float cscale = sc2;
#pragma unroll
        for (int kc = 0; kc < 2; ++kc)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int m = 16 * kc + 2 * c4 + (j & 1) + 8 * (j >> 1);
                rope_cs_s(rsm, m, pos0, cs[kc][j], sn[kc][j]);
                cs[kc][j] *= cscale;
                sn[kc][j] *= cscale;
            }
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            float x[4][4];                        // [kc][j]: dims 16kc + {2c4, 2c4+1, 2c4+8, 2c4+9}
#pragma unroll
            for (int kc = 0; kc < 4; ++kc) {
                const unsigned u0 = qraw[half][kc][0];
                const unsigned u1 = qraw[half][kc][1];
                x[kc][0] = __uint_as_float(u0 << 16); x[kc][1] = __uint_as_float(u0 & 0xffff0000u);
                x[kc][2] = __uint_as_float(u1 << 16); x[kc][3] = __uint_as_float(u1 & 0xffff0000u);
            }
            if (half == 1) {
#pragma unroll
                for (int kc = 0; kc < 2; ++kc)
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int m = 16 * kc + 2 * c4 + (j & 1) + 8 * (j >> 1);
                        const float c8 = rsm.c8[m], s8 = rsm.s8[m];
                        const float cn = cs[kc][j] * c8 - sn[kc][j] * s8;
                        sn[kc][j] = sn[kc][j] * c8 + cs[kc][j] * s8;
                        cs[kc][j] = cn;
                    }
            }
#pragma unroll
            for (int kc = 0; kc < 2; ++kc) {      // pair (dim m in kc, dim m+32 in kc+2)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float xa = x[kc][j], xb = x[kc + 2][j];
                    x[kc][j] = xa * cs[kc][j] - xb * sn[kc][j];
                    x[kc + 2][j] = xb * cs[kc][j] + xa * sn[kc][j];
                    qmax = fmaxf(qmax, fmaxf(fabsf(x[kc][j]), fabsf(x[kc + 2][j])));
                }
            }
#pragma unroll
            for (int kc = 0; kc < 4; ++kc) {
                qa[kc][half] = pack_f16(x[kc][0], x[kc][1]);          // a0 / a1: k = 2c4, 2c4+1
                qa[kc][2 + half] = pack_f16(x[kc][2], x[kc][3]);      // a2 / a3: k = 2c4+8, 2c4+9
                if constexpr (SAVE) {
                    const float u = 1.f / sc2;
                    qs[kc][half] = pack_bf16(x[kc][0] * u, x[kc][1] * u);
                    qs[kc][2 + half] = pack_bf16(x[kc][2] * u, x[kc][3] * u);
                }
            }
        }
    }
    if (qmax >= 65520.f) raise_status(a.status, kStatusRange);
    const int qlo = bw + g4, qhi = bw + g4 + 8;   // absolute queries of this thread's rows
    const bool vlo = qlo < s.T && g4 < kRowsPerWarp;
    const bool vhi = qhi < s.T && g4 + 8 < kRowsPerWarp;
    // a rung slot of a row is attended when d_k <= query; this lane takes part
    // in a row's rung softmax only where it holds part of the row's score
    const float qlo_eff = (contrib && vlo) ? (float)qlo : -1.f;
    const float qhi_eff = (contrib && vhi) ? (float)qhi : -1.f;
    const size_t rowbase = (size_t)bh * s.T;
    if constexpr (SAVE) {
        // rotated query rows 0..14 of the warp's tile, through the warp's stage
        // (16-byte chunk c of row r at chunk c ^ r) and out as runs of rows
        static_assert(TEAMS == 1, "the residuals are written by the one-head form");
        unsigned* stage = ostage[warp];
        __nv_bfloat16* QT = reinterpret_cast<__nv_bfloat16*>(a.res_qt) + rowbase * kHeadDim;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
#pragma unroll
            for (int kc = 0; kc < 4; ++kc) {
                stage[g4 * 32 + (((2 * kc) ^ g4) << 2) + c4] = qs[kc][half];
                stage[g4 * 32 + (((2 * kc + 1) ^ g4) << 2) + c4] = qs[kc][2 + half];
            }
            __syncwarp();
            const int nrow = min(half ? kRowsPerWarp - 8 : 8, s.T - (bw + 8 * half));
#pragma unroll
            for (int c = lane; c < 64; c += 32) {
                const int r = c >> 3, ch = c & 7;
                if (r < nrow) {
                    const uint4 v = *reinterpret_cast<const uint4*>(stage + r * 32 + ((ch ^ r) << 2));
                    *reinterpret_cast<uint4*>(QT + (size_t)(bw + 8 * half + r) * kHeadDim + 8 * ch) = v;
                }
            }
            __syncwarp();                         // the stage is read before it is rewritten
        }
    }

    // The active rungs in increasing d: those with d_k > bw + 14 are masked
    // for every row of the warp and form the tail of the list.
    int n_use = L.n_act;
    while (n_use > 0 && L.act_d[n_use - 1] > (float)(bw + kRowsPerWarp - 1)) --n_use;

    const bool ok_k = mbar_wait(&bars[0], 0);

    // ---- window band scores: keys [bw - Wp, bw + 16), n-tile j covers 8 keys
    float sw[NT][4];
    {
        const int rb = L.win_smem + wrel - Wp + lr;
        const unsigned ab = sbase + ((unsigned)rb << 7) + ((unsigned)((rb ^ lh) & 7) << 4);
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            unsigned b0, b1, b2, b3;
            ldsm_x4(ab + 1024u * j, b0, b1, b2, b3);
            mma_f16_16816_z(sw[j], qa[0], b0, b1);
            mma_f16_16816(sw[j], qa[1], b2, b3);
            ldsm_x4((ab ^ 64u) + 1024u * j, b0, b1, b2, b3);
            mma_f16_16816(sw[j], qa[2], b0, b1);
            mma_f16_16816(sw[j], qa[3], b2, b3);
        }
    }
    float mlo = -INFINITY, mhi = -INFINITY;       // per-lane partial maxima until every slot is in
    {
        const int tb = g4 + Wp - 2 * c4;          // distance query - key of entry (row g4, column 2c4) in n-tile 0
#pragma unroll
        for (int j = 0; j < NT; ++j)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int t = tb + (e >= 2 ? 8 : 0) - 8 * j - (e & 1);
                if ((unsigned)t > (unsigned)s.W) sw[j][e] = -INFINITY;
            }
        if (bw < Wp) {                            // the first tile: columns before position 0
#pragma unroll
            for (int j = 0; j < NT; ++j)
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (8 * j + 2 * c4 + (e & 1) < Wp - bw) sw[j][e] = -INFINITY;
        }
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            mlo = fmaxf(mlo, fmaxf(sw[j][0], sw[j][1]));
            mhi = fmaxf(mhi, fmaxf(sw[j][2], sw[j][3]));
        }
    }

    // ---- rung scores (log2 units) of the rows this lane takes part in
    const float inv_sc2 = 1.f / sc2;
    // SAVE: the residual arrays of this head, addressed by 32-bit offsets
    // (S T <= 33 x 2^20 with W, K <= 16 and T <= 2^20); row qhi = qlo + 8 is 8
    // entries on
    float* Pg = SAVE ? a.res_P + (size_t)bh * a.S * s.T : nullptr;   // residual exp(s - max) per slot
    float* SDg = SAVE ? a.res_sd + (size_t)bh * a.r.K * s.T : nullptr;
    float rs[kMmaMaxRungs][2];
    // rung i of the list sorted by d (i < n_use)
    auto score_rung = [&](int i) {
        const int r = L.act_smem[i] + wrel + lr;
        const unsigned ak = sbase + ((unsigned)r << 7) + ((unsigned)((r ^ lh) & 7) << 4);
        float s0[4], s1[4];
        unsigned b0, b1, b2, b3;
        ldsm_x4(ak, b0, b1, b2, b3);
        mma_f16_16816_z(s0, qa[0], b0, b1);
        mma_f16_16816(s0, qa[1], b2, b3);
        ldsm_x4(ak + 1024u, b0, b1, b2, b3);
        mma_f16_16816_z(s1, qa[0], b0, b1);
        mma_f16_16816(s1, qa[1], b2, b3);
        ldsm_x4(ak ^ 64u, b0, b1, b2, b3);
        mma_f16_16816(s0, qa[2], b0, b1);
        mma_f16_16816(s0, qa[3], b2, b3);
        ldsm_x4((ak ^ 64u) + 1024u, b0, b1, b2, b3);
        mma_f16_16816(s1, qa[2], b0, b1);
        mma_f16_16816(s1, qa[3], b2, b3);
        const float w = L.act_w[i];
        const float c0 = fmaf(ib0, w, ia0), c1 = fmaf(ib1, w, ia1), c7 = fmaf(-m7, w, m7);
        float plo = fmaf(c0, s0[0], fmaf(c1, s0[1], c7 * s1[0]));
        float phi = fmaf(c0, s1[2], c1 * s1[3]);
        plo += __shfl_sync(0xffffffffu, plo, src);
        phi += __shfl_sync(0xffffffffu, phi, src);
        const float d = L.act_d[i];
        rs[i][0] = d <= qlo_eff ? plo : -INFINITY;
        rs[i][1] = d <= qhi_eff ? phi : -INFINITY;
        mlo = fmaxf(mlo, rs[i][0]);
        mhi = fmaxf(mhi, rs[i][1]);
        if constexpr (SAVE) {
            float sdl = fmaf(ib0, s0[0], fmaf(ib1, s0[1], -m7 * s1[0]));
            float sdh = fmaf(ib0, s1[2], ib1 * s1[3]);
            sdl += __shfl_sync(0xffffffffu, sdl, src);
            sdh += __shfl_sync(0xffffffffu, sdh, src);
            if (writer) {
                float* sd = SDg + (unsigned)(L.act_k[i] * s.T + qlo);
                if (vlo) sd[0] = sdl * inv_sc2;
                if (vhi) sd[8] = sdh * inv_sc2;
            }
        }
    };
#pragma unroll
    for (int i = 0; i < kMmaMaxRungs; ++i) {
        if (i >= n_use) break;
        score_rung(i);
    }

    if (TEAMS == 1) {
        // ---- the last warp done with the keys stages the values into the same
        // buffer (acquire-release counter: every warp's key reads come before
        // the copies; the others go on without waiting)
        asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
        __syncwarp();
        unsigned before = 0;
        if (lane == 0) before = atom_add_acq_rel(&keys_done, 1u);
        before = __shfl_sync(0xffffffffu, before, 0);
        if (before == kWarps - 1) {
            asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
            issue_rows(buf, &tmV.m64, &tmV.m8, L, i0, head, &bars[1], lane);
        }
    }

    // ---- probabilities (unnormalised, row max -> exactly 1) while values arrive
    mlo = quad_max(mlo);
    mhi = quad_max(mhi);
    if (mlo == -INFINITY) mlo = 0.f;              // rows beyond T: keep arithmetic finite
    if (mhi == -INFINITY) mhi = 0.f;
    unsigned pa[NT][2];                           // window band P as bf16 A fragments
    // SAVE: entry (j, e) of the band is row g4 + 8 (e >> 1), slot
    // t = tb + 8 (e >> 1) - 8 j - (e & 1), at offset t T + bw + row
    const int tb = g4 + Wp - 2 * c4;
    const int pband = tb * s.T + bw + g4;
#pragma unroll
    for (int j = 0; j < NT; ++j) {
        const float e0 = ex2(sw[j][0] - mlo), e1 = ex2(sw[j][1] - mlo);
        const float e2 = ex2(sw[j][2] - mhi), e3 = ex2(sw[j][3] - mhi);
        pa[j][0] = pack_bf16(e0, e1);
        pa[j][1] = pack_bf16(e2, e3);
        if constexpr (SAVE) {                     // window slot t of rows 0..14 (0 before position 0)
            const float ev[4] = {e0, e1, e2, e3};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const bool hi = e >= 2;
                const int dt = (hi ? 8 : 0) - 8 * j - (e & 1);
                const int t = tb + dt;
                if ((hi ? vhi : vlo) && (unsigned)t <= (unsigned)s.W)
                    Pg[(unsigned)(pband + dt * s.T + (hi ? 8 : 0))] = ev[e];
            }
        }
    }

    if constexpr (SAVE) {
        // ---- residual p of the active rungs no row of the warp attends (the
        // tail of the list sorted by d): 0
        if (c4 == 0) {
            for (int i = n_use; i < L.n_act; ++i) {
                float* row = Pg + (unsigned)((s.W + 1 + L.act_k[i]) * s.T + qlo);
                if (vlo) row[0] = 0.f;
                if (vhi) row[8] = 0.f;
            }
        }
    }

    // rung probabilities (and their residuals) while the values arrive: the
    // rung scores become p = 2^(s - max) in place
#pragma unroll
    for (int i = 0; i < kMmaMaxRungs; ++i) {
        if (i >= n_use) break;
        rs[i][0] = ex2(rs[i][0] - mlo);           // 0 when masked
        rs[i][1] = ex2(rs[i][1] - mhi);
        if constexpr (SAVE) {
            if (writer) {                         // residual p of the rung
                float* row = Pg + (unsigned)((s.W + 1 + L.act_k[i]) * s.T + qlo);
                if (vlo) row[0] = rs[i][0];
                if (vhi) row[8] = rs[i][1];
            }
        }
    }

    const bool ok_v = mbar_wait(&bars[1], 0);

    // o: the value product; osum: the row sums of the same rounded weights
    float o[8][4], osum[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int n = 0; n < 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;

    // ---- window band values: k-chunks of 16 keys (+ one of 8 when NT is odd)
    {
        const int rv = L.win_smem + wrel - Wp + lv;
        const unsigned av = vbase + ((unsigned)rv << 7) + ((unsigned)((rv ^ lq) & 7) << 4);
#pragma unroll
        for (int kk = 0; kk + 1 < NT; kk += 2) {
            const unsigned afr[4] = {pa[kk][0], pa[kk][1], pa[kk + 1][0], pa[kk + 1][1]};
#pragma unroll
            for (int n = 0; n < 8; n += 2) {
                unsigned b0, b1, b2, b3;
                ldsm_x4_t((av ^ (unsigned)(n << 4)) + 1024u * kk, b0, b1, b2, b3);
                mma_bf16_16816(o[n], afr, b0, b1);
                mma_bf16_16816(o[n + 1], afr, b2, b3);
            }
            mma_bf16_16816(osum, afr, kOnesBf16x2, kOnesBf16x2);
        }
    }
    if constexpr (NT & 1) {
        const int kk = NT - 1;
        const int rt = L.win_smem + wrel - Wp + 8 * kk + lr;
        const unsigned at = vbase + ((unsigned)rt << 7) + ((unsigned)((rt ^ lh) & 7) << 4);
#pragma unroll
        for (int n = 0; n < 8; n += 4) {
            unsigned b0, b1, b2, b3;
            ldsm_x4_t(at ^ (unsigned)(n << 4), b0, b1, b2, b3);
            mma_bf16_1688(o[n], pa[kk][0], pa[kk][1], b0);
            mma_bf16_1688(o[n + 1], pa[kk][0], pa[kk][1], b1);
            mma_bf16_1688(o[n + 2], pa[kk][0], pa[kk][1], b2);
            mma_bf16_1688(o[n + 3], pa[kk][0], pa[kk][1], b3);
        }
        mma_bf16_1688(osum, pa[kk][0], pa[kk][1], kOnesBf16x2);
    }

    // ---- rung values: Phat[r][x] = p_r w at x = r, p_r (1-w) at x = r + 1
    // A-fragment columns of this thread: 2c4 + {0,1} (a0, a1) and 2c4 + 8 + {0,1} (a2, a3).
    auto value_rung = [&](int i) {
        const float w = L.act_w[i];
        const float plo = rs[i][0], phi = rs[i][1];
        // Phat in bf16 (a1, row g4+8 at columns 2c4.., is zero); the row sums
        // come from the same rounded entries (the ones product below)
        const float c0 = fmaf(ib0, w, ia0), c1 = fmaf(ib1, w, ia1), c7 = fmaf(-m7, w, m7);
        const unsigned ahi[4] = {pack_bf16(c0 * plo, c1 * plo), 0u, pack_bf16(c7 * plo, 0.f),
                                 pack_bf16(c0 * phi, c1 * phi)};
        const int rv = L.act_smem[i] + wrel + lv;
        const unsigned av = vbase + ((unsigned)rv << 7) + ((unsigned)((rv ^ lq) & 7) << 4);
#pragma unroll
        for (int n = 0; n < 8; n += 2) {
            unsigned b0, b1, b2, b3;
            ldsm_x4_t(av ^ (unsigned)(n << 4), b0, b1, b2, b3);
            mma_bf16_16816(o[n], ahi, b0, b1);
            mma_bf16_16816(o[n + 1], ahi, b2, b3);
        }
        mma_bf16_16816(osum, ahi, kOnesBf16x2, kOnesBf16x2);
    };
#pragma unroll
    for (int i = 0; i < kMmaMaxRungs; ++i) {
        if (i >= n_use) break;
        value_rung(i);
    }

    // ---- normalise and store rows 0..14 of the tile
    const float llo = osum[0], lhi = osum[2];     // every column of the ones product is the row sum
    const bool ok = ok_k && ok_v;
    if (!ok) raise_status(a.status, kStatusWaitTimeout);
    const float inv_lo = ok ? 1.f / llo : __int_as_float(0x7fc00000);
    const float inv_hi = ok ? 1.f / lhi : __int_as_float(0x7fc00000);
    // Rows g4 (half 0) and g4 + 8 (half 1) leave through this warp's stage, 8
    // rows of 128 bytes at a time (16-byte chunk c of row r at chunk c ^ r), and
    // go out as runs of consecutive rows: 512 contiguous bytes per warp store.
    __nv_bfloat16* O = reinterpret_cast<__nv_bfloat16*>(a.out) + rowbase * kHeadDim;
    if constexpr (TEAMS == 1) {
        unsigned* stage = ostage[warp];
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const float inv = half ? inv_hi : inv_lo;
#pragma unroll
            for (int n = 0; n < 8; ++n)
                stage[g4 * 32 + ((n ^ g4) << 2) + c4] = pack_bf16(o[n][2 * half] * inv, o[n][2 * half + 1] * inv);
            __syncwarp();
            // rows bw + 8 half + r, r < 8 (7 in the second half: row 15 of the
            // tile is the next warp's), below T
            const int nrow = min(half ? kRowsPerWarp - 8 : 8, s.T - (bw + 8 * half));
#pragma unroll
            for (int c = lane; c < 64; c += 32) {
                const int r = c >> 3, ch = c & 7;
                if (r < nrow) {
                    const uint4 v = *reinterpret_cast<const uint4*>(stage + r * 32 + ((ch ^ r) << 2));
                    *reinterpret_cast<uint4*>(O + (size_t)(bw + 8 * half + r) * kHeadDim + 8 * ch) = v;
                }
            }
            __syncwarp();                             // the stage is read before it is rewritten
        }
    } else {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            if (!(half ? vhi : vlo)) continue;
            const float inv = half ? inv_hi : inv_lo;
            __nv_bfloat16* row = O + (size_t)(half ? qhi : qlo) * kHeadDim;
#pragma unroll
            for (int n = 0; n < 8; ++n)
                *reinterpret_cast<unsigned*>(row + 8 * n + 2 * c4) =
                    pack_bf16(o[n][2 * half] * inv, o[n][2 * half + 1] * inv);
        }
    }
    // (a timed-out wait leaves NaN in lse and 1 / row sum too)
    if (c4 == 0 && vlo) {
        a.lse[(size_t)bh * s.T + qlo] = ok ? (mlo + __log2f(llo)) * kLn2 : inv_lo;
        if constexpr (SAVE) a.res_il[(size_t)bh * s.T + qlo] = inv_lo;
    }
    if (c4 == 0 && vhi) {
        a.lse[(size_t)bh * s.T + qhi] = ok ? (mhi + __log2f(lhi)) * kLn2 : inv_hi;
        if constexpr (SAVE) a.res_il[(size_t)bh * s.T + qhi] = inv_hi;
    }
    }                                             // query heads of the group
}

// ------------------------------------------------------------ host side ----

template <int NT, int TEAMS>
cudaError_t launch_nt(const RowMaps& mk, const RowMaps& mv, const FwdArgs& a, const MmaLayout& L,
                      unsigned grid, size_t smem, cudaStream_t st) {
    // (the grouped form runs only without residuals)
    auto kern = a.res_P ? fwd_mma_kernel<NT, TEAMS, TEAMS == 1> : fwd_mma_kernel<NT, TEAMS, false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_kernel(kern, dim3(grid), dim3(kWarps * 32 * TEAMS), smem, st, mk, mv, a, L);
}

}  // namespace

static PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess && q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

bool encode_rows_map(CUtensorMap* map, const void* base, CUtensorMapDataType dt, int T, int heads, int box_rows) {
    auto fn = get_encode();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)kHeadDim, (cuuint64_t)T, (cuuint64_t)heads};
    cuuint64_t strides[2] = {(cuuint64_t)kHeadDim * 2, (cuuint64_t)T * kHeadDim * 2};
    cuuint32_t box[3] = {(cuuint32_t)kHeadDim, (cuuint32_t)box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(map, dt, 3, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

size_t fwd_mma_smem_bytes(const MmaLayout& L) { return (size_t)L.buf_rows * 128 + 1024; }

// the barriers and counter of a CTA (rounded up), its warps' output stages
// and the RoPE steps
size_t fwd_mma_static_smem() { return 64 + kWarps * 1024 + sizeof(RopeSmem); }

size_t fwd_mma_gqa_smem_limit() { return 227 * 1024 - 64 - 1024; }

namespace {

struct Iv { int a, b; };

// Merge relative row intervals (sorted by start), round each merged interval up
// to whole 8-row TMA boxes and lay them out one after another in shared memory.
// An interval that starts before the rounded end of the one before it joins it:
// the rounded intervals then cover disjoint relative rows, so every relative
// row has exactly one shared row and a slab is contiguous in shared memory.
void layout_intervals(Iv* iv, int n, MmaLayout* L) {
    for (int i = 1; i < n; ++i)                   // insertion sort by start
        for (int j = i; j > 0 && iv[j].a < iv[j - 1].a; --j) { Iv t = iv[j]; iv[j] = iv[j - 1]; iv[j - 1] = t; }
    int m = 0;
    for (int i = 0; i < n; ++i) {
        const int end8 = m > 0 ? iv[m - 1].a + (((iv[m - 1].b - iv[m - 1].a) + 7) & ~7) : 0;
        if (m > 0 && iv[i].a < end8) { if (iv[i].b > iv[m - 1].b) iv[m - 1].b = iv[i].b; }
        else iv[m++] = iv[i];
    }
    L->n_iv = m;
    int rows = 0;
    for (int i = 0; i < m; ++i) {
        const int len = ((iv[i].b - iv[i].a) + 7) & ~7;      // whole 8-row TMA boxes
        L->iv_start[i] = iv[i].a;
        L->iv_len[i] = len;
        L->iv_smem[i] = rows;
        rows += len;
    }
    L->rows = rows;
}

int smem_row_of(const MmaLayout& L, int rel) {
    for (int i = 0; i < L.n_iv; ++i)
        if (rel >= L.iv_start[i] && rel < L.iv_start[i] + L.iv_len[i]) return L.iv_smem[i] + (rel - L.iv_start[i]);
    return -1;
}

int interval_of(const MmaLayout& L, int smem_row) {
    for (int i = 0; i < L.n_iv; ++i)
        if (smem_row >= L.iv_smem[i] && smem_row < L.iv_smem[i] + L.iv_len[i]) return i;
    return 0;
}

// Active rungs sorted by d (ties by index), with their shared rows and the
// merged interval of each slab.
void active_list(const RungParams& r, MmaLayout* L) {
    L->n_act = 0;
    for (int i = 0; i < kMmaMaxRungs; ++i) {
        L->act_k[i] = 0; L->act_s0[i] = 0; L->act_smem[i] = 0; L->act_w[i] = 0.f; L->act_d[i] = 3.0e38f;
    }
    for (int k = 0; k < r.K; ++k) {
        if (!((r.active >> k) & 1u)) continue;
        int i = L->n_act++;
        while (i > 0 && L->act_d[i - 1] > r.d[k]) {
            L->act_k[i] = L->act_k[i - 1]; L->act_s0[i] = L->act_s0[i - 1]; L->act_smem[i] = L->act_smem[i - 1];
            L->act_w[i] = L->act_w[i - 1]; L->act_d[i] = L->act_d[i - 1];
            --i;
        }
        L->act_k[i] = k; L->act_s0[i] = r.s0[k]; L->act_smem[i] = L->rung_smem[k];
        L->act_w[i] = r.w[k]; L->act_d[i] = r.d[k];
    }
    for (int i = 0; i < kMmaMaxRungs; ++i) L->act_iv[i] = i < L->n_act ? interval_of(*L, L->act_smem[i]) : 0;
    L->win_iv = interval_of(*L, L->win_smem);
}

void rope_steps(double rope_base, MmaLayout* L) {
    for (int m = 0; m < kHalf; ++m) {
        const double theta = std::pow(rope_base, -2.0 * m / (double)kHeadDim);
        L->rope_c8[m] = (float)std::cos(8.0 * theta);
        L->rope_s8[m] = (float)std::sin(8.0 * theta);
    }
}

}  // namespace

// Copy boxes in issue order (per interval: 64-row boxes, then 8-row boxes);
// split them at the first box that starts at or after the tile regions.
void plan_tile_regions(MmaLayout* L, int reserve_rows) {
    L->buf_rows = L->rows > reserve_rows ? L->rows : reserve_rows;
    L->lo_start = L->rows;
    L->bytes_lo = 0;
    L->bytes_hi = 0;
    for (int iv = 0; iv < L->n_iv; ++iv) {
        int r = 0;
        auto box = [&](int srow, int h) {
            if (srow >= reserve_rows) {
                if (srow < L->lo_start) L->lo_start = srow;
                L->bytes_lo += (unsigned)h * 128u;
            } else {
                L->bytes_hi += (unsigned)h * 128u;
            }
        };
        for (; r + 64 <= L->iv_len[iv]; r += 64) box(L->iv_smem[iv] + r, 64);
        for (; r < L->iv_len[iv]; r += 8) box(L->iv_smem[iv] + r, 8);
    }
}

bool build_mma_layout(const Shape& s, const RungParams& r, double rope_base, size_t smem_limit, MmaLayout* L,
                      int reserve_rows) {
    if (s.W > 16 || r.K > kMmaMaxRungs) return false;
    const int NT = s.W == 0 ? 2 : (s.W <= 8 ? 3 : 4);
    const int Wp = NT * 8 - 16;
    L->nt = NT;
    // relative rows each warp tile reads; the tile spans rows [0, kMmaTile + 1)
    Iv iv[kMmaMaxRungs + 1];
    int n = 0;
    iv[n++] = {-Wp, kMmaTile + 1};
    for (int k = 0; k < r.K; ++k)
        if ((r.active >> k) & 1u) iv[n++] = {-r.s0[k] - 1, kMmaTile + 1 - r.s0[k]};
    layout_intervals(iv, n, L);
    L->win_smem = smem_row_of(*L, 0);
    rope_steps(rope_base, L);
    for (int k = 0; k < kMmaMaxRungs; ++k) L->rung_smem[k] = 0;
    for (int k = 0; k < r.K; ++k)
        if ((r.active >> k) & 1u) L->rung_smem[k] = smem_row_of(*L, -r.s0[k] - 1);
    active_list(r, L);
    L->buf_rows = L->rows;
    L->lo_start = 0;
    L->bytes_lo = (unsigned)L->rows * 128u;
    L->bytes_hi = 0;
    if (reserve_rows > 0) plan_tile_regions(L, reserve_rows);
    return fwd_mma_smem_bytes(*L) <= smem_limit;
}

bool build_key_layout(const Shape& s, const RungParams& r, double rope_base, size_t smem_limit, MmaLayout* L) {
    if (s.W > 16 || r.K > kMmaMaxRungs) return false;
    const int NT = s.W == 0 ? 2 : (s.W <= 8 ? 3 : 4);
    const int Wp = NT * 8 - 16;
    L->nt = NT;
    // query rows, relative to the first key of the tile, that a key tile's
    // warps read: the band [0, kMmaTile + 1 + Wp) and per rung the slab
    // [s0, s0 + kMmaTile + 1) (near query j + s0 and far query j + s0 + 1)
    Iv iv[kMmaMaxRungs + 1];
    int n = 0;
    iv[n++] = {0, kMmaTile + 1 + Wp};
    for (int k = 0; k < r.K; ++k)
        if ((r.active >> k) & 1u) iv[n++] = {r.s0[k], r.s0[k] + kMmaTile + 1};
    layout_intervals(iv, n, L);
    L->win_smem = smem_row_of(*L, 0);
    rope_steps(rope_base, L);
    for (int k = 0; k < kMmaMaxRungs; ++k) L->rung_smem[k] = 0;
    for (int k = 0; k < r.K; ++k)
        if ((r.active >> k) & 1u) L->rung_smem[k] = smem_row_of(*L, r.s0[k]);
    active_list(r, L);
    L->buf_rows = L->rows;
    L->lo_start = 0;
    L->bytes_lo = (unsigned)L->rows * 128u;
    L->bytes_hi = 0;
    return fwd_mma_smem_bytes(*L) <= smem_limit;
}

cudaError_t launch_fwd_mma(const FwdArgs& a, const MmaLayout& L, cudaStream_t st) {
    const long long tiles = (a.s.T + kMmaTile - 1) / kMmaTile;
    RowMaps mk, mv;
    const int heads = a.s.B * a.s.Hkv;
    if (tiles * a.s.B * a.s.H <= 0) return cudaSuccess;
    if (!encode_row_maps(&mk, a.kt, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, a.s.T, heads) ||
        !encode_row_maps(&mv, a.v, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.s.T, heads))
        return cudaErrorInvalidValue;
    // Grouped-query attention: one CTA per kv head's tile with both staged
    // tensors resident, when they fit and no residuals are written (with the
    // residual stores, one CTA per query head's tile with two CTAs per SM
    // measured faster; L2 then serves the group's repeated row reads).
    const size_t smem2 = 2 * (size_t)L.rows * 128 + 1024;
    if (a.s.G >= 2 && smem2 <= fwd_mma_gqa_smem_limit() && !a.res_P) {
        const unsigned grid = (unsigned)(tiles * heads);
        switch (L.nt) {
        case 2: return launch_nt<2, 2>(mk, mv, a, L, grid, smem2, st);
        case 3: return launch_nt<3, 2>(mk, mv, a, L, grid, smem2, st);
        default: return launch_nt<4, 2>(mk, mv, a, L, grid, smem2, st);
        }
    }
    const unsigned grid = (unsigned)(tiles * a.s.B * a.s.H);
    const size_t smem = fwd_mma_smem_bytes(L);
    switch (L.nt) {
    case 2: return launch_nt<2, 1>(mk, mv, a, L, grid, smem, st);
    case 3: return launch_nt<3, 1>(mk, mv, a, L, grid, smem, st);
    default: return launch_nt<4, 1>(mk, mv, a, L, grid, smem, st);
    }
}

}  // namespace fibattn
