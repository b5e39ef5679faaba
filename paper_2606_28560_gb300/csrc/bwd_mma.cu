// bwd_mma.cu -- query-centric backward on tensor cores (mma.sync, m16n8) with
// TMA staging: the chain rule of the attended-set forward (arXiv 2606.28560,
// Section 2 "Attended set" and "Implementation note").
//
// Tiles and staged rows are those of the tensor-core forward: a warp owns a
// 16-row tile of queries placed every 15 queries, a CTA the union of rows its
// tiles read (window band and one 16-row slab per rung).  With
// Delta_i = dO_i . o_i (the forward output), the gradient of every score is
// known as soon as its slot is:  dS = p (dp - Delta),  p = exp(s - lse),
// dp = dO . val.  So the backward needs each staged tensor once:
//
//   values staged (bf16):  dP = dO V^T     window band 16 x (16+Wp) and the
//                          16 x 16 slab of each rung; a rung keeps its far and
//                          floor columns: dp = (1-w) dp0 + w dp1, ddp = dp1 - dp0
//   keys staged (fp16):    S = Q~ K~^T     same blocks; p, dS per slot, then
//                          dq~ += dS_band K~_band + dShat_k K~_slab
//                          with dShat_k[u][u] = dS w, dShat_k[u][u+1] = dS (1-w)
//
// and the rung-distance gradient of query i (row -1 is a zero row):
//   dL/dd_k += p (scale (s1 - s0)(dp - Delta) + ddp)
// with s1, s0 the raw far and floor dot products.  p and dS per slot (zero
// where not attended; slot-major arrays [head][slot][T], so that the key pass
// reads runs of consecutive queries), Delta and the rotated queries go to the
// workspace for the key-centric pass (the rotated queries as bf16).
//
// Range: dS enters the dq MMAs as fp16 (11-bit significand, the type of the
// staged rotated keys), whose normal range (6.1e-5 .. 65504) is far narrower
// than bf16's.  Each query row's dS is therefore multiplied by a power of two
// c before the rounding, chosen from the row's largest |dp - Delta| (a bound
// on |dS|, p <= 1) so that the scaled values reach [2^14, 2^15); the row's
// dq~ is divided by c at the end (exact, a power of two).  So no row's score
// gradients underflow or overflow fp16 whatever the magnitude of dO (a
// bf16-autocast training step passes upstream gradients of 1e-5 .. 1e-8).
// Accumulation is fp32.
#include <cmath>
#include <type_traits>

#include "fibattn_internal.cuh"
#include "fwd_mma.cuh"
#include "mma_common.cuh"

namespace fibattn {
namespace {

using namespace mma;

constexpr float kLog2e = 1.4426950408889634f;
constexpr int kWarps = kMmaWarps;
constexpr int kRowsPerWarp = 15;

__device__ __forceinline__ float bf_lo(unsigned u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf_hi(unsigned u) { return __uint_as_float(u & 0xffff0000u); }

// Biased fp32 exponent of the power of two c with m c in [2^14, 2^15), for
// m = a row's largest |dp - Delta| (c = 1 for m = 0 or subnormal; clamped so
// that both c and 1 / c are normal).
__device__ __forceinline__ int ds_scale_exp(float m) {
    const int e = (__float_as_int(m) >> 23) & 0xff;
    return e == 0 ? 127 : min(253, max(1, 268 - e));
}
__device__ __forceinline__ float exp_to_f(int ce) { return __int_as_float(ce << 23); }

// DD: also the rung-distance gradient dL/dd_k (off when the caller asks for
// neither dtheta nor dd, e.g. a fixed alpha schedule).
// SV: p of every slot (stored unnormalised, with 1 / row sum per query) and
// the far-minus-floor rung scores come from the forward's residuals (p and the
// rotated queries serve the key pass too), so
// the scores are not recomputed: dS = p (dp - Delta) is formed in the value
// phase and the key phase only accumulates dq~.
template <int NT, bool DD, bool SV>
__global__ void __launch_bounds__(kWarps * 32, 2)
bwd_query_mma_kernel(const __grid_constant__ RowMaps tmK, const __grid_constant__ RowMaps tmV,
                     const __grid_constant__ QTileMaps tm, BwdArgs a, MmaLayout L) {
    grid_dependency_sync();
    constexpr int Wp = NT * 8 - 16;
    extern __shared__ unsigned char smem_raw[];
    __shared__ unsigned long long bars[4];        // V (first batch), K~, V (second batch), tile rows
    // !SV: rung dp, ddp of each warp's tile rows.  SV: p (replaced by dS once
    // known) and sd (replaced by the row's dL/dd_k term once known) of each
    // active rung (list order) and tile row.
    constexpr int kXs = SV ? 2 * kMmaMaxRungs * kMmaTile : kWarps * kMmaMaxRungs * 16 * 2;
    __shared__ __align__(16) float xs[kXs];
    auto dps = reinterpret_cast<float (*)[kMmaMaxRungs][16][2]>(xs);
    auto psd = reinterpret_cast<float (*)[kMmaMaxRungs][kMmaTile]>(xs);
    __shared__ float gsm[kWarps][kMmaMaxRungs];           // per-warp rung-gradient sums
    __shared__ unsigned long long kbar[kMmaMaxRungs + 1]; // key rows of each merged interval
    __shared__ unsigned rel_cnt[kMmaMaxRungs + 1];        // warps done with an interval's value rows
    unsigned char* buf = reinterpret_cast<unsigned char*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const unsigned sbase = smem_u32(buf);

    const Shape& s = a.s;
    const int bh = (int)fdiv(blockIdx.x, s.dTiles);              // block = bh * tiles + tile
    const int i0 = ((int)blockIdx.x - bh * (int)s.dTiles.d) * kMmaTile;
    const int b = (int)fdiv((unsigned)bh, s.dH), hk = (int)fdiv((unsigned)(bh - b * s.H), s.dG);
    const int head = b * s.Hkv + hk;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g4 = lane >> 2, c4 = lane & 3;
    const int wrel = warp * kRowsPerWarp;
    const int bw = i0 + wrel;

    // ---- the tile's q, dO, o rows (two 64-row boxes each) to buffer rows
    // [0, 384), and the value rows that do not overlap them
    __shared__ RopeSmem rsm;
    rope_to_smem(rsm, a.rope, L, tid);
    if (tid == 0) {
        for (int i = 0; i < 4; ++i) mbar_init(&bars[i], 1);
        for (int j = 0; j < L.n_iv; ++j) {
            mbar_init(&kbar[j], 1);
            rel_cnt[j] = 0u;
        }
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    if (warp == 0) {
        __syncwarp();
        if (lane == 0) {
            mbar_expect_tx(&bars[3], (SV ? 2u : 3u) * 128u * 128u);
            const CUtensorMap* maps[3] = {&tm.q, &tm.g, &tm.o};
#pragma unroll
            for (int t = SV ? 1 : 0; t < 3; ++t)
#pragma unroll
                for (int hb = 0; hb < 2; ++hb)
                    tma_load_3d(buf + (size_t)(128 * t + 64 * hb) * 128, maps[t], 0, i0 + 64 * hb, bh, &bars[3]);
        }
        if (L.bytes_lo) issue_rows_batch(buf, &tmV.m64, &tmV.m8, L, i0, head, &bars[0], lane, false);
    }

    const int qlo = bw + g4, qhi = bw + g4 + 8;
    const bool vlo = qlo < s.T && g4 < kRowsPerWarp;
    const bool vhi = qhi < s.T && g4 + 8 < kRowsPerWarp;
    const size_t rowbase = (size_t)bh * s.T;
    float* Pg = a.Ps + (size_t)bh * a.S * s.T;       // [slot][T] of this head
    float* DSg = a.DSs + (size_t)bh * a.S * s.T;

    // SV: the residual (unnormalised) p of the window band at this thread's
    // accumulator entries and 1 / (row sum) of its rows (registers), and p
    // and sd of the active rungs for the tile's rows (shared memory, 4-byte
    // asynchronous copies by every thread); p = residual p / row sum
    float pb[NT][4];
    float il_lo = 0.f, il_hi = 0.f;
    if constexpr (SV) {
        il_lo = vlo ? a.res_il[rowbase + qlo] : 0.f;
        il_hi = vhi ? a.res_il[rowbase + qhi] : 0.f;
#pragma unroll
        for (int j = 0; j < NT; ++j)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const bool hi = e >= 2;
                const int r = hi ? g4 + 8 : g4;
                const int t = r + Wp - (8 * j + 2 * c4 + (e & 1));
                pb[j][e] = ((hi ? vhi : vlo) && t >= 0 && t <= s.W) ? Pg[(unsigned)(t * s.T + bw + r)] : 0.f;
            }
        const float* SDg = DD ? a.res_sd + (size_t)bh * a.r.K * s.T : nullptr;
        for (int u = tid; u < L.n_act * kMmaTile; u += kWarps * 32) {
            const int i = u / kMmaTile, r = u - i * kMmaTile;
            const bool in = i0 + r < s.T;
            const int q = in ? i0 + r : 0, k = L.act_k[i];
            cp_async4(&psd[0][i][r], Pg + (size_t)(s.W + 1 + k) * s.T + q, in);
            if (DD) cp_async4(&psd[1][i][r], SDg + (size_t)k * s.T + q, in);
        }
        asm volatile("cp.async.commit_group;\n" ::: "memory");
    }

    __syncthreads();                              // barrier init visible
    bool ok_v = mbar_wait(&bars[3], 0);

    // A fragments of this warp's 16 tile rows from a staged region: for
    // k-chunk kc, registers (row g4, dims 16kc + 2c4..), (row g4+8, same),
    // (row g4, dims 16kc + 8 + 2c4..), (row g4+8, same)
    auto tile_frags = [&](int region, unsigned (&f)[4][4]) {
        const int row = 128 * region + wrel + (lane & 7) + 8 * ((lane >> 3) & 1);
#pragma unroll
        for (int kc = 0; kc < 4; ++kc)
            ldsm_x4(row_chunk(sbase, row, 2 * kc + (lane >> 4)), f[kc][0], f[kc][1], f[kc][2], f[kc][3]);
    };

    // ---- dO as bf16 A fragments; Delta = dO . o of rows g4, g4+8
    unsigned da[4][4];
    float dlt_lo, dlt_hi;
    {
        unsigned oa[4][4];
        tile_frags(1, da);
        tile_frags(2, oa);
        float part[2] = {0.f, 0.f};
#pragma unroll
        for (int kc = 0; kc < 4; ++kc)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                part[j & 1] = fmaf(bf_lo(da[kc][j]), bf_lo(oa[kc][j]), part[j & 1]);
                part[j & 1] = fmaf(bf_hi(da[kc][j]), bf_hi(oa[kc][j]), part[j & 1]);
            }
        dlt_lo = quad_sum(part[0]);
        dlt_hi = quad_sum(part[1]);
    }

    // ---- q~ as fp16 A fragments (RoPE pairs m, m+32 in the same thread), and
    // as bf16 for the key pass (qs)
    unsigned qa[4][4], qs[SV ? 1 : 4][4];
    if constexpr (!SV) {
        float qmax = 0.f;                         // largest |q~| of the thread: fp16 holds < 65520
        unsigned qr[4][4];
        tile_frags(0, qr);
        float cs[2][4], sn[2][4];
#pragma unroll
        for (int kc = 0; kc < 2; ++kc)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int m = 16 * kc + 2 * c4 + (j & 1) + 8 * (j >> 1);
                rope_cs_s(rsm, m, qlo, cs[kc][j], sn[kc][j]);
            }
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            float x[4][4];
#pragma unroll
            for (int kc = 0; kc < 4; ++kc) {
                const unsigned u0 = qr[kc][half], u1 = qr[kc][2 + half];
                x[kc][0] = bf_lo(u0); x[kc][1] = bf_hi(u0);
                x[kc][2] = bf_lo(u1); x[kc][3] = bf_hi(u1);
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
            for (int kc = 0; kc < 2; ++kc) {
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
                qa[kc][half] = pack_f16(x[kc][0], x[kc][1]);
                qa[kc][2 + half] = pack_f16(x[kc][2], x[kc][3]);
                qs[kc][half] = pack_bf16(x[kc][0], x[kc][1]);
                qs[kc][2 + half] = pack_bf16(x[kc][2], x[kc][3]);
            }
        }
        if (qmax >= 65520.f) raise_status(a.status, kStatusRange);
    }
    // ---- q~ rows to the workspace (for the key pass): written in place of the
    // staged q rows, then stored by TMA (rows past T are clipped); the value
    // rows of the second batch follow once the store has read them.  (SV: the
    // forward wrote them; the second batch follows once the tile rows are read.)
    if constexpr (SV) {
        asm volatile("cp.async.wait_group 0;\n" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
    }
    __syncthreads();                              // every warp has read the tile rows (SV: residuals landed)
    if constexpr (!SV) {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            if (g4 + 8 * half >= kRowsPerWarp) continue;
            const int row = wrel + g4 + 8 * half;
#pragma unroll
            for (int kc = 0; kc < 4; ++kc) {
                asm volatile("st.shared.b32 [%0], %1;\n" :: "r"(row_chunk(sbase, row, 2 * kc) + 4 * c4), "r"(qs[kc][half]));
                asm volatile("st.shared.b32 [%0], %1;\n" :: "r"(row_chunk(sbase, row, 2 * kc + 1) + 4 * c4),
                             "r"(qs[kc][2 + half]));
            }
        }
        asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
        __syncthreads();
    }
    if (warp == 0) {
        if (!SV && lane == 0) {
#pragma unroll
            for (int t = 0; t < 3; ++t)                // 3 boxes of 40 rows: the tile's 120 queries
                asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];\n"
                             :: "l"(&tm.qt), "r"(0), "r"(i0 + 40 * t), "r"(bh),
                                "r"(sbase + (unsigned)(40 * t * 128)) : "memory");
            asm volatile("cp.async.bulk.commit_group;\n" ::: "memory");
            asm volatile("cp.async.bulk.wait_group.read 0;\n" ::: "memory");
        }
        __syncwarp();
        issue_rows_batch(buf, &tmV.m64, &tmV.m8, L, i0, head, &bars[2], lane, true);
    }
    const float lse2_lo = (!SV && vlo) ? a.lse[rowbase + qlo] * kLog2e : 0.f;
    const float lse2_hi = (!SV && vhi) ? a.lse[rowbase + qhi] * kLog2e : 0.f;

    // Columns of a rung slab: row r's far row is x = r (weight w), its floor
    // row x = r+1 (weight 1-w).  Of this thread's accumulator and A-fragment
    // entries (rows g4, g4+8; columns 2c4, 2c4+1 and 2c4+8, 2c4+9) only those
    // with x - r in {-1, 0, 1} can be either, a pattern fixed by
    // delta = 2c4 - g4: entries (g4, 2c4 + u) and (g4+8, 2c4+8 + u) take the
    // interpolation weights  u=0: w if delta = 0, 1-w if delta = 1;
    //                        u=1: w if delta = -1, 1-w if delta = 0,
    // each weight of the form A + B w; the far-minus-floor difference takes
    // +1 / -1 at the same places.  Row g4 = 7 also has its floor at column 8.
    const int dl = 2 * c4 - g4;
    const float ia0 = dl == 1 ? 1.f : 0.f, ib0 = dl == 0 ? 1.f : (dl == 1 ? -1.f : 0.f);
    const float ia1 = dl == 0 ? 1.f : 0.f, ib1 = dl == -1 ? 1.f : (dl == 0 ? -1.f : 0.f);
    const float df0 = dl == 0 ? 1.f : (dl == 1 ? -1.f : 0.f), df1 = dl == -1 ? 1.f : (dl == 0 ? -1.f : 0.f);
    const float m7 = (g4 == 7 && c4 == 0) ? 1.f : 0.f;

    // Value rows: the first batch (rows from L.lo_start on) now, the second
    // before the first use of a row below L.lo_start.
    if (L.bytes_lo) ok_v = mbar_wait(&bars[0], 0) && ok_v;
    bool hi_done = false;
    auto need_rows = [&](int row) {
        if (!hi_done && row < L.lo_start) {
            ok_v = mbar_wait(&bars[2], 0) && ok_v;
            hi_done = true;
        }
    };
    need_rows(L.win_smem + wrel - Wp);

    // ---- window band dp = dO . v
    float dpw[NT][4];
    {
        const unsigned ab = row_chunk(sbase, L.win_smem + wrel - Wp + (lane & 7), lane >> 3);
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            unsigned b0, b1, b2, b3;
            ldsm_x4(ab + 1024u * j, b0, b1, b2, b3);
            mma_bf16_16816_z(dpw[j], da[0], b0, b1);
            mma_bf16_16816(dpw[j], da[1], b2, b3);
            ldsm_x4((ab ^ 64u) + 1024u * j, b0, b1, b2, b3);
            mma_bf16_16816(dpw[j], da[2], b0, b1);
            mma_bf16_16816(dpw[j], da[3], b2, b3);
        }
    }
    // the rows' largest |dp - Delta| over the band (rung terms join below):
    // the bound on |dS| that sets the rows' fp16 scale
    float emax_lo = 0.f, emax_hi = 0.f;
#pragma unroll
    for (int j = 0; j < NT; ++j) {
        emax_lo = fmaxf(emax_lo, fmaxf(fabsf(dpw[j][0] - dlt_lo), fabsf(dpw[j][1] - dlt_lo)));
        emax_hi = fmaxf(emax_hi, fmaxf(fabsf(dpw[j][2] - dlt_hi), fabsf(dpw[j][3] - dlt_hi)));
    }
    emax_lo = quad_max(emax_lo);
    emax_hi = quad_max(emax_hi);
    // window band dS = p (dp - Delta) (SV: here, kept in fp32 until the rows'
    // scale is known; else in the key phase, once the scores are known); dS
    // per slot to the workspace
    unsigned dsa[NT][2];
    float dsb[SV ? NT : 1][4];
    if constexpr (SV) {
#pragma unroll
        for (int j = 0; j < NT; ++j) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const bool hi = e >= 2;
                const int r = hi ? g4 + 8 : g4;
                const int t = r + Wp - (8 * j + 2 * c4 + (e & 1));
                dsb[j][e] = pb[j][e] * (hi ? il_hi : il_lo) * (dpw[j][e] - (hi ? dlt_hi : dlt_lo));
                if ((hi ? vhi : vlo) && t >= 0 && t <= s.W) DSg[(unsigned)(t * s.T + bw + r)] = dsb[j][e];
            }
        }
    }
    // Rungs in increasing d; those masked for every row of the warp's tile
    // (d > bw + 14) form the tail of the list.
    int n_use = 0;
    while (n_use < L.n_act && L.act_d[n_use] <= (float)(bw + kRowsPerWarp - 1)) ++n_use;

    // Key rows replace the value rows interval by interval.  A warp visits
    // intervals in decreasing order (the band's is the last; a rung with larger
    // d sits lower) and releases each one as it moves below it; the last of the
    // kWarps warps to release an interval issues its key copies.
    int rel = L.n_iv;                             // intervals >= rel are released
    auto release_above = [&](int iv) {
        while (rel - 1 > iv) {
            const int j = --rel;
            if (L.iv_smem[j] < L.lo_start) need_rows(-1);   // second value batch landed first
            asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
            __syncwarp();
            if (lane == 0 && atom_add_acq_rel(&rel_cnt[j], 1u) == kWarps - 1)
                issue_interval(buf, &tmK.m64, &tmK.m8, L, j, i0, head, &kbar[j]);
            __syncwarp();
        }
    };

    // ---- rung dp (interpolated) and ddp = dp_far - dp_floor, to shared memory
    if constexpr (SV) {
        // Two rungs per iteration (their MMA and reduction chains are
        // independent), the last of an odd count alone.  Each lane tracks its
        // row's largest |dp - Delta| (lanes c4 < 2: row g4, else g4 + 8).
        float emax_row = 0.f;
        // per rung: this lane's shares of dp and ddp for rows g4 and g4+8,
        // reduce-scattered over the quad (lanes c4 = 0, 1 end with row g4,
        // lanes 2, 3 with row g4+8); lanes 0 and 2 then form their row's dS
        // (from the residual p) and dL/dd_k term, the terms summed over the
        // warp's rows in a fixed order; dS replaces p in shared memory for
        // the key phase
        const bool up = c4 >= 2;
        const int row = wrel + g4 + (up ? 8 : 0);
        const bool rv = up ? vhi : vlo;
        auto value_block = [&](int i, auto nu) {  // NU rungs from list position i
            constexpr int NU = decltype(nu)::value;
            release_above(L.act_iv[i]);
#pragma unroll
            for (int u = 0; u < NU; ++u) need_rows(L.act_smem[i + u] + wrel);
            float dt[NU][2][4];
#pragma unroll
            for (int u = 0; u < NU; ++u) {
                const unsigned ak = row_chunk(sbase, L.act_smem[i + u] + wrel + (lane & 7), lane >> 3);
#pragma unroll
                for (int t = 0; t < 2; ++t) {
                    unsigned b0, b1, b2, b3;
                    ldsm_x4(ak + 1024u * t, b0, b1, b2, b3);
                    mma_bf16_16816_z(dt[u][t], da[0], b0, b1);
                    mma_bf16_16816(dt[u][t], da[1], b2, b3);
                    ldsm_x4((ak ^ 64u) + 1024u * t, b0, b1, b2, b3);
                    mma_bf16_16816(dt[u][t], da[2], b0, b1);
                    mma_bf16_16816(dt[u][t], da[3], b2, b3);
                }
            }
            float ds[NU];
            [[maybe_unused]] float gr[NU];
#pragma unroll
            for (int u = 0; u < NU; ++u) {
                const float w = L.act_w[i + u], w1 = 1.f - w;
                const float c0 = fmaf(ib0, w, ia0), c1 = fmaf(ib1, w, ia1), c7 = m7 * w1;
                const float x0 = fmaf(c0, dt[u][0][0], fmaf(c1, dt[u][0][1], c7 * dt[u][1][0]));
                const float x2 = fmaf(c0, dt[u][1][2], c1 * dt[u][1][3]);
                float x1 = 0.f, x3 = 0.f;
                if constexpr (DD) {
                    x1 = fmaf(df0, dt[u][0][0], fmaf(df1, dt[u][0][1], -m7 * dt[u][1][0]));
                    x3 = fmaf(df0, dt[u][1][2], df1 * dt[u][1][3]);
                }
                float dp = up ? x2 : x0;
                [[maybe_unused]] float ddp = up ? x3 : x1;
                dp += __shfl_xor_sync(0xffffffffu, up ? x0 : x2, 2);
                if constexpr (DD) ddp += __shfl_xor_sync(0xffffffffu, up ? x1 : x3, 2);
                dp += __shfl_xor_sync(0xffffffffu, dp, 1);
                if constexpr (DD) ddp += __shfl_xor_sync(0xffffffffu, ddp, 1);
                const float p = rv ? psd[0][i + u][row] * (up ? il_hi : il_lo) : 0.f;
                const float e = dp - (up ? dlt_hi : dlt_lo);
                emax_row = fmaxf(emax_row, fabsf(e));
                ds[u] = p * e;
                if constexpr (DD) {               // the row's dL/dd_k term, summed over the tile at the end
                    const float sd = rv ? psd[1][i + u][row] : 0.f;
                    gr[u] = p * fmaf(s.scale * sd, e, ddp);
                }
            }
            __syncwarp();                         // the quad has read p (and sd) before they are replaced
            if ((c4 & 1) == 0 && rv) {
#pragma unroll
                for (int u = 0; u < NU; ++u) {
                    psd[0][i + u][row] = ds[u];
                    if constexpr (DD) psd[1][i + u][row] = gr[u];
                    DSg[(unsigned)((s.W + 1 + L.act_k[i + u]) * s.T + bw + g4 + (up ? 8 : 0))] = ds[u];
                }
            }
        };
        int i = 0;
#pragma unroll 1
        for (; i + 1 < n_use; i += 2) value_block(i, std::integral_constant<int, 2>{});
        if (i < n_use) value_block(i, std::integral_constant<int, 1>{});
        emax_lo = fmaxf(emax_lo, __shfl_sync(0xffffffffu, emax_row, lane & ~3));
        emax_hi = fmaxf(emax_hi, __shfl_sync(0xffffffffu, emax_row, (lane & ~3) | 2));
    } else {
    #pragma unroll 1
        for (int i = 0; i < n_use; ++i) {
            release_above(L.act_iv[i]);
            const float w = L.act_w[i], w1 = 1.f - w;
            need_rows(L.act_smem[i] + wrel);
            float dt[2][4];
    #pragma unroll
            for (int t = 0; t < 2; ++t) {
                dt[t][0] = dt[t][1] = dt[t][2] = dt[t][3] = 0.f;
                const int krow = L.act_smem[i] + wrel + 8 * t + (lane & 7);
    #pragma unroll
                for (int kc = 0; kc < 4; kc += 2) {
                    unsigned b0, b1, b2, b3;
                    ldsm_x4(row_chunk(sbase, krow, 2 * kc + (lane >> 3)), b0, b1, b2, b3);
                    mma_bf16_16816(dt[t], da[kc], b0, b1);
                    mma_bf16_16816(dt[t], da[kc + 1], b2, b3);
                }
            }
            const float c0 = fmaf(ib0, w, ia0), c1 = fmaf(ib1, w, ia1), c7 = m7 * w1;
            // this lane's shares of dp and ddp for rows g4 and g4+8
            const float x0 = fmaf(c0, dt[0][0], fmaf(c1, dt[0][1], c7 * dt[1][0]));
            const float x2 = fmaf(c0, dt[1][2], c1 * dt[1][3]);
            float x1 = 0.f, x3 = 0.f;
            if constexpr (DD) {
                x1 = fmaf(df0, dt[0][0], fmaf(df1, dt[0][1], -m7 * dt[1][0]));
                x3 = fmaf(df0, dt[1][2], df1 * dt[1][3]);
            }
            const float dp_lo = quad_sum(x0), dp_hi = quad_sum(x2);
            const float ddp_lo = DD ? quad_sum(x1) : 0.f, ddp_hi = DD ? quad_sum(x3) : 0.f;
            emax_lo = fmaxf(emax_lo, fabsf(dp_lo - dlt_lo));
            emax_hi = fmaxf(emax_hi, fabsf(dp_hi - dlt_hi));
            if (c4 == 0) {
                *reinterpret_cast<float2*>(dps[warp][i][g4]) = make_float2(dp_lo, ddp_lo);
                *reinterpret_cast<float2*>(dps[warp][i][g4 + 8]) = make_float2(dp_hi, ddp_hi);
            }
        }
    }
    release_above(-1);

    // the rows' fp16 scale c (a power of two) and 1 / c
    const int ce_lo = ds_scale_exp(emax_lo), ce_hi = ds_scale_exp(emax_hi);
    const float cs_lo = exp_to_f(ce_lo), cs_hi = exp_to_f(ce_hi);
    if constexpr (SV) {
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            dsa[j][0] = pack_f16(dsb[j][0] * cs_lo, dsb[j][1] * cs_lo);
            dsa[j][1] = pack_f16(dsb[j][2] * cs_hi, dsb[j][3] * cs_hi);
        }
    }

    // key rows of an interval: waited for before its first use
    bool ok_k = true;
    unsigned waited = 0u;
    auto need_keys = [&](int iv) {
        if (!((waited >> iv) & 1u)) {
            ok_k = mbar_wait(&kbar[iv], 0) && ok_k;
            waited |= 1u << iv;
        }
    };

    const float sc2 = s.scale * kLog2e;

    float dq[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n) dq[n][0] = dq[n][1] = dq[n][2] = dq[n][3] = 0.f;

    // ---- window band: scores, p, dS; P and dS per slot to the workspace (SV:
    // dS is known); dq~ += dS_band K~_band
    need_keys(L.win_iv);
    if constexpr (SV) __syncwarp();               // dS of the value phase, written by the quad's lane 0
    if constexpr (!SV) {
        float sw[NT][4];
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            sw[j][0] = sw[j][1] = sw[j][2] = sw[j][3] = 0.f;
            const int krow = L.win_smem + wrel - Wp + 8 * j + (lane & 7);
#pragma unroll
            for (int kc = 0; kc < 4; kc += 2) {
                unsigned b0, b1, b2, b3;
                ldsm_x4(row_chunk(sbase, krow, 2 * kc + (lane >> 3)), b0, b1, b2, b3);
                mma_f16_16816(sw[j], qa[kc], b0, b1);
                mma_f16_16816(sw[j], qa[kc + 1], b2, b3);
            }
        }
#pragma unroll
        for (int j = 0; j < NT; ++j) {
            float dsv[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const bool hi = e >= 2;
                const int r = hi ? g4 + 8 : g4;
                const int n = 8 * j + 2 * c4 + (e & 1);
                const int t = r + Wp - n;                     // distance query - key
                const int key = bw - Wp + n;
                const bool rv = hi ? vhi : vlo;
                const bool inband = t >= 0 && t <= s.W;
                const bool ok = rv && inband && key >= 0;
                const float p = ok ? exp2f(sw[j][e] * sc2 - (hi ? lse2_hi : lse2_lo)) : 0.f;
                dsv[e] = p * (dpw[j][e] - (hi ? dlt_hi : dlt_lo));
                if (rv && inband) {
                    Pg[(size_t)t * s.T + bw + r] = p;
                    DSg[(size_t)t * s.T + bw + r] = dsv[e];
                }
            }
            dsa[j][0] = pack_f16(dsv[0] * cs_lo, dsv[1] * cs_lo);
            dsa[j][1] = pack_f16(dsv[2] * cs_hi, dsv[3] * cs_hi);
        }
    }
    {
        const unsigned avb = row_chunk(sbase, L.win_smem + wrel - Wp + (lane & 7) + (lane & 8), lane >> 4);
#pragma unroll
        for (int kk = 0; kk + 1 < NT; kk += 2) {
            const unsigned afr[4] = {dsa[kk][0], dsa[kk][1], dsa[kk + 1][0], dsa[kk + 1][1]};
#pragma unroll
            for (int n = 0; n < 8; n += 2) {
                unsigned b0, b1, b2, b3;
                ldsm_x4_t((avb ^ (unsigned)(n << 4)) + 1024u * kk, b0, b1, b2, b3);
                mma_f16_16816(dq[n], afr, b0, b1);
                mma_f16_16816(dq[n + 1], afr, b2, b3);
            }
        }
        if constexpr (NT & 1) {
            const int kk = NT - 1;
            const unsigned at = row_chunk(sbase, L.win_smem + wrel - Wp + 8 * kk + (lane & 7), lane >> 3);
#pragma unroll
            for (int n = 0; n < 8; n += 4) {
                unsigned b0, b1, b2, b3;
                ldsm_x4_t(at ^ (unsigned)(n << 4), b0, b1, b2, b3);
                mma_f16_1688(dq[n], dsa[kk][0], dsa[kk][1], b0);
                mma_f16_1688(dq[n + 1], dsa[kk][0], dsa[kk][1], b1);
                mma_f16_1688(dq[n + 2], dsa[kk][0], dsa[kk][1], b2);
                mma_f16_1688(dq[n + 3], dsa[kk][0], dsa[kk][1], b3);
            }
        }
    }

    // ---- rungs that no row of the tile attends: zero slots for the key pass
    for (int i = n_use; i < L.n_act; ++i) {
        const int slot = s.W + 1 + L.act_k[i];
        if (c4 == 0) {                            // (SV: the forward wrote p = 0 there)
            const unsigned o = (unsigned)(slot * s.T + qlo);
            if (vlo) { if (!SV) Pg[o] = 0.f; DSg[o] = 0.f; }
            if (vhi) { if (!SV) Pg[o + 8] = 0.f; DSg[o + 8] = 0.f; }
        }
        if constexpr (SV) {
            if (DD && lane < kRowsPerWarp) psd[1][i][wrel + lane] = 0.f;   // no dL/dd_k term
        } else {
            if (lane == 0) gsm[warp][L.act_k[i]] = 0.f;
        }
    }
    // ---- rungs: scores, p, dS, dL/dd_k (SV: dS from the value phase);
    // dq~ += dShat_k K~_slab.  SV: two rungs per iteration (the second's dS
    // loads and fragments overlap the first's products); the odd last rung
    // goes through the loop below.
    int i_first = 0;
    if constexpr (SV) {
#pragma unroll 1
        for (; i_first + 1 < n_use; i_first += 2) {
            need_keys(L.act_iv[i_first]);
            need_keys(L.act_iv[i_first + 1]);
            unsigned afr2[2][4];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int ii = i_first + u;
                const float w = L.act_w[ii], w1 = 1.f - w;
                const float c0 = fmaf(ib0, w, ia0), c1 = fmaf(ib1, w, ia1), c7 = m7 * w1;
                const float dsl = vlo ? psd[0][ii][wrel + g4] * cs_lo : 0.f;
                const float dsh = vhi ? psd[0][ii][wrel + g4 + 8] * cs_hi : 0.f;
                afr2[u][0] = pack_f16(c0 * dsl, c1 * dsl);
                afr2[u][1] = 0u;
                afr2[u][2] = pack_f16(c7 * dsl, 0.f);
                afr2[u][3] = pack_f16(c0 * dsh, c1 * dsh);
            }
            const int lv = (lane & 7) + (lane & 8);
            const unsigned av0 = row_chunk(sbase, L.act_smem[i_first] + wrel + lv, lane >> 4);
            const unsigned av1 = row_chunk(sbase, L.act_smem[i_first + 1] + wrel + lv, lane >> 4);
#pragma unroll
            for (int n = 0; n < 8; n += 2) {
                unsigned b0, b1, b2, b3, e0, e1, e2, e3;
                ldsm_x4_t(av0 ^ (unsigned)(n << 4), b0, b1, b2, b3);
                ldsm_x4_t(av1 ^ (unsigned)(n << 4), e0, e1, e2, e3);
                mma_f16_16816(dq[n], afr2[0], b0, b1);
                mma_f16_16816(dq[n + 1], afr2[0], b2, b3);
                mma_f16_16816(dq[n], afr2[1], e0, e1);
                mma_f16_16816(dq[n + 1], afr2[1], e2, e3);
            }
        }
    }
#pragma unroll 1
    for (int i = i_first; i < n_use; ++i) {
        need_keys(L.act_iv[i]);
        const float w = L.act_w[i], w1 = 1.f - w;
        const float c0 = fmaf(ib0, w, ia0), c1 = fmaf(ib1, w, ia1), c7 = m7 * w1;
        float ds_lo, ds_hi;
        if constexpr (SV) {
            ds_lo = vlo ? psd[0][i][wrel + g4] : 0.f;
            ds_hi = vhi ? psd[0][i][wrel + g4 + 8] : 0.f;
        } else {
            const int k = L.act_k[i];
            const int slot = s.W + 1 + k;
            float st[2][4];
#pragma unroll
            for (int t = 0; t < 2; ++t) {
                st[t][0] = st[t][1] = st[t][2] = st[t][3] = 0.f;
                const int krow = L.act_smem[i] + wrel + 8 * t + (lane & 7);
#pragma unroll
                for (int kc = 0; kc < 4; kc += 2) {
                    unsigned b0, b1, b2, b3;
                    ldsm_x4(row_chunk(sbase, krow, 2 * kc + (lane >> 3)), b0, b1, b2, b3);
                    mma_f16_16816(st[t], qa[kc], b0, b1);
                    mma_f16_16816(st[t], qa[kc + 1], b2, b3);
                }
            }
            // interpolated score and far-minus-floor raw score of rows g4, g4+8
            const float si_lo = quad_sum(fmaf(c0, st[0][0], fmaf(c1, st[0][1], c7 * st[1][0])));
            const float si_hi = quad_sum(fmaf(c0, st[1][2], c1 * st[1][3]));
            const float dk = L.act_d[i];
            const bool okl = vlo && dk <= (float)qlo, okh = vhi && dk <= (float)qhi;
            const float2 dpl = *reinterpret_cast<const float2*>(dps[warp][i][g4]);
            const float2 dph = *reinterpret_cast<const float2*>(dps[warp][i][g4 + 8]);
            const float dp_lo = dpl.x, ddp_lo = dpl.y, dp_hi = dph.x, ddp_hi = dph.y;
            const float p_lo = okl ? exp2f(si_lo * sc2 - lse2_lo) : 0.f;
            const float p_hi = okh ? exp2f(si_hi * sc2 - lse2_hi) : 0.f;
            const float e_lo = dp_lo - dlt_lo, e_hi = dp_hi - dlt_hi;
            ds_lo = p_lo * e_lo;
            ds_hi = p_hi * e_hi;
            if (c4 == 0) {
                if (vlo) { Pg[(size_t)slot * s.T + qlo] = p_lo; DSg[(size_t)slot * s.T + qlo] = ds_lo; }
                if (vhi) { Pg[(size_t)slot * s.T + qhi] = p_hi; DSg[(size_t)slot * s.T + qhi] = ds_hi; }
            }
            if constexpr (DD) {
                // far-minus-floor raw scores; dL/dd_k of this warp's rows, in a fixed order over the rows
                const float sd_lo = quad_sum(fmaf(df0, st[0][0], fmaf(df1, st[0][1], -m7 * st[1][0])));
                const float sd_hi = quad_sum(fmaf(df0, st[1][2], df1 * st[1][3]));
                float g = 0.f;
                if (c4 == 0)
                    g = p_lo * fmaf(s.scale * sd_lo, e_lo, ddp_lo) + p_hi * fmaf(s.scale * sd_hi, e_hi, ddp_hi);
                g += __shfl_xor_sync(0xffffffffu, g, 4);
                g += __shfl_xor_sync(0xffffffffu, g, 8);
                g += __shfl_xor_sync(0xffffffffu, g, 16);
                if (lane == 0) gsm[warp][k] = g;
            }
        }

        // dShat_k as fp16 A fragment: the interpolation weights times the row's
        // scaled dS
        const float dsl = ds_lo * cs_lo, dsh = ds_hi * cs_hi;
        const unsigned afr[4] = {pack_f16(c0 * dsl, c1 * dsl), 0u, pack_f16(c7 * dsl, 0.f),
                                 pack_f16(c0 * dsh, c1 * dsh)};
        const unsigned av = row_chunk(sbase, L.act_smem[i] + wrel + (lane & 7) + (lane & 8), lane >> 4);
#pragma unroll
        for (int n = 0; n < 8; n += 2) {
            unsigned b0, b1, b2, b3;
            ldsm_x4_t(av ^ (unsigned)(n << 4), b0, b1, b2, b3);
            mma_f16_16816(dq[n], afr, b0, b1);
            mma_f16_16816(dq[n + 1], afr, b2, b3);
        }
    }

    // ---- dq = R(-theta pos) scale dq~, rows 0..14 of the tile
    const bool ok = ok_k && ok_v;
    if (!ok) raise_status(a.status, kStatusWaitTimeout);
    // scale / c of each row (exact: c is a power of two)
    const float sc_lo = ok ? s.scale * exp_to_f(254 - ce_lo) : __int_as_float(0x7fc00000);
    const float sc_hi = ok ? s.scale * exp_to_f(254 - ce_hi) : __int_as_float(0x7fc00000);
    __nv_bfloat16* dQ = reinterpret_cast<__nv_bfloat16*>(a.dq) + rowbase * kHeadDim;
    // cos, sin of pair m = 8n + 2c4 + u (m + 32 sits in n-tile n + 4) at qlo,
    // then advanced by 8 positions for qhi with the host's cos, sin(8 theta_m)
    float ec[4][2], es[4][2];
#pragma unroll
    for (int n = 0; n < 4; ++n)
#pragma unroll
        for (int u = 0; u < 2; ++u) rope_cs_s(rsm, 8 * n + 2 * c4 + u, qlo, ec[n][u], es[n][u]);
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        if (half == 1) {
#pragma unroll
            for (int n = 0; n < 4; ++n)
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int m = 8 * n + 2 * c4 + u;
                    const float c8 = rsm.c8[m], s8 = rsm.s8[m];
                    const float cn = ec[n][u] * c8 - es[n][u] * s8;
                    es[n][u] = es[n][u] * c8 + ec[n][u] * s8;
                    ec[n][u] = cn;
                }
        }
        if (!(half ? vhi : vlo)) continue;
        const int q = half ? qhi : qlo;
        const float sc = half ? sc_hi : sc_lo;
        __nv_bfloat16* row = dQ + (size_t)q * kHeadDim;
#pragma unroll
        for (int n = 0; n < 4; ++n) {
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const float xa = dq[n][2 * half + u] * sc, xb = dq[n + 4][2 * half + u] * sc;
                dq[n][2 * half + u] = xa * ec[n][u] + xb * es[n][u];
                dq[n + 4][2 * half + u] = xb * ec[n][u] - xa * es[n][u];
            }
        }
#pragma unroll
        for (int n = 0; n < 8; ++n)
            *reinterpret_cast<unsigned*>(row + 8 * n + 2 * c4) = pack_bf16(dq[n][2 * half], dq[n][2 * half + 1]);
    }

    // ---- per-CTA rung partials, summed in a fixed order
    if constexpr (DD && SV) {
        // the tile rows' terms of active rung i are in psd[1][i][0..119] (0
        // for rows past T and rungs a warp does not attend): warp w sums list
        // entries 2w and 2w+1 (lane l: rows l, l+32, l+64, l+96, then a
        // butterfly over the lanes); inactive rungs get a zero partial
        __syncthreads();
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int i = 2 * warp + u;
            if (i >= L.n_act) break;
            float x = 0.f;
#pragma unroll
            for (int r = lane; r < kMmaTile; r += 32) x += psd[1][i][r];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
            if (lane == 0) a.rpart[(size_t)L.act_k[i] * a.nblk_q + blockIdx.x] = __float2ll_rn(x * 4294967296.0f);
        }
        if (tid < a.r.K && !((a.r.active >> tid) & 1u)) a.rpart[(size_t)tid * a.nblk_q + blockIdx.x] = 0;
    } else if constexpr (DD) {                    // warps summed in a fixed order
        __syncthreads();
        float x = 0.f;
        if (tid < a.r.K && ((a.r.active >> tid) & 1u))
            for (int wv = 0; wv < kWarps; ++wv) x += gsm[wv][tid];
        write_rung_partials(a, x);
    }
    // ---- no copy may outlive the CTA: the key rows of intervals that no rung
    // of this warp read were issued (by the last warp to release them) but not
    // waited for, and the rotated-query store may still be writing
    for (int j = 0; j < L.n_iv; ++j) need_keys(j);
    if (!SV && tid == 0) asm volatile("cp.async.bulk.wait_group 0;\n" ::: "memory");
}

template <int NT>
cudaError_t launch_nt(const RowMaps& mk, const RowMaps& mv, const QTileMaps& mt, const BwdArgs& a,
                      const MmaLayout& L, unsigned grid, size_t smem, cudaStream_t st) {
    auto kern = a.saved ? (a.want_dd ? bwd_query_mma_kernel<NT, true, true> : bwd_query_mma_kernel<NT, false, true>)
                        : (a.want_dd ? bwd_query_mma_kernel<NT, true, false> : bwd_query_mma_kernel<NT, false, false>);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_kernel(kern, dim3(grid), dim3(kWarps * 32), smem, st, mk, mv, mt, a, L);
}

}  // namespace

size_t bwd_mma_static_smem() {
    // dps, gsm, the interval barriers and counters, the four phase barriers, the RoPE steps
    return sizeof(float) * kWarps * kMmaMaxRungs * 16 * 2 + sizeof(float) * kWarps * kMmaMaxRungs +
           (sizeof(unsigned long long) + sizeof(unsigned)) * (kMmaMaxRungs + 1) + 4 * sizeof(unsigned long long) +
           sizeof(RopeSmem) + 64;
}

int bwd_mma_blocks(const Shape& s) {
    const long long tiles = (s.T + kMmaTile - 1) / kMmaTile;
    return (int)(tiles * s.B * s.H);
}

cudaError_t launch_bwd_query_mma(const BwdArgs& a, const MmaLayout& L, cudaStream_t st) {
    const long long grid = bwd_mma_blocks(a.s);
    if (grid <= 0) return cudaSuccess;
    RowMaps mk, mv;
    QTileMaps mt;
    const int heads = a.s.B * a.s.Hkv, qheads = a.s.B * a.s.H;
    if (!encode_row_maps(&mk, a.kt, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, a.s.T, heads) ||
        !encode_row_maps(&mv, a.v, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.s.T, heads) ||
        !encode_rows_map(&mt.q, a.q, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.s.T, qheads, 64) ||
        !encode_rows_map(&mt.g, a.dout, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.s.T, qheads, 64) ||
        !encode_rows_map(&mt.o, a.out, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.s.T, qheads, 64) ||
        !encode_rows_map(&mt.qt, a.qt, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.s.T, qheads, 40))
        return cudaErrorInvalidValue;
    const size_t smem = fwd_mma_smem_bytes(L);
    switch (L.nt) {
    case 2: return launch_nt<2>(mk, mv, mt, a, L, (unsigned)grid, smem, st);
    case 3: return launch_nt<3>(mk, mv, mt, a, L, (unsigned)grid, smem, st);
    default: return launch_nt<4>(mk, mv, mt, a, L, (unsigned)grid, smem, st);
    }
}

}  // namespace fibattn
