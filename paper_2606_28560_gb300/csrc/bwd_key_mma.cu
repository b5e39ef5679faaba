// bwd_key_mma.cu -- key-centric backward on tensor cores (mma.sync, m16n8)
// with TMA staging (arXiv 2606.28560, Section 2 "Attended set"; the chain
// rule of the forward).
//
// Key row j receives, from each query head of its group, the slots that read
// it: window slot t of query j + t (weight 1), rung k of query j + s0_k (its
// floor row, weight 1 - w_k) and of query j + s0_k + 1 (its far row, weight w_k):
//   dv_j  = sum c p dO_i,        dk~_j = scale sum c dS q~_i,
// with p and dS = p (dp - Delta) per (query, slot) from the tensor-core query
// pass (slot-major arrays, read as runs of consecutive queries).  A warp owns 16 keys (tiles every 15 keys, the 16th row discarded);
// with the keys as MMA rows and the queries as the reduction index both sums
// are products of a banded matrix with staged query rows:
//   window band  acc += P_band^T  X[b, b+16+Wp)       P_band^T[r][x] = p(b+x, t = x-r)
//   rung k       acc += Phat_k^T  X[b+s0, b+s0+16)    Phat_k^T[r][r] = (1-w) p, [r][r+1] = w p
// with X = dO rows (bf16, pass 0: dv) and then X = q~ rows (bf16, pass 1:
// dk~, dS in place of p).  The CTA stages the union of the query rows its
// warps read, one tensor (and query head) at a time, in one buffer.
// A-operand values: p and dS as bf16 (the exponent range of fp32: no score
// gradient underflows, however small the upstream gradient); accumulation
// fp32.  A warp's dv
// and dk rows leave through its rung table as runs of consecutive rows.
#include <cmath>

#include "fibattn_internal.cuh"
#include "fwd_mma.cuh"
#include "mma_common.cuh"

namespace fibattn {
namespace {

using namespace mma;

constexpr int kWarps = kMmaWarps;
constexpr int kRowsPerWarp = 15;

// One staged tensor of one query head: accumulate banded A x staged rows.
// X: p or dS of this query head, slot-major [S][T]; operands bf16.
// IL (p from the forward residuals, unnormalised): 1 / (row sum) per query
// of this head; the warp copies the entries its values need into its rung
// table and its band strip (wil, 32 floats) and scales each value.
template <int NT>
__device__ __forceinline__ void key_pass(float (&acc)[8][4], const float* X, const BwdArgs& a, const MmaLayout& L,
                                         unsigned sbase, int bw, int wrel, int g4, int c4, int lane, bool vlo,
                                         bool vhi, unsigned long long* bar, unsigned parity, bool& ok,
                                         float (*rv)[16], const float* IL = nullptr, float* wil = nullptr) {
    const Shape& s = a.s;
    if (IL) {                                     // 1 / row sum of the queries the values below belong to
#pragma unroll
        for (int j = 0; j < kMmaMaxRungs * 16 / 32; ++j) {
            const int u = lane + 32 * j;
            const int i = u >> 4, x = u & 15;
            const int q = bw + L.act_s0[i] + x;
            const bool use = i < L.n_act && q < s.T;
            cp_async4(&rv[i][x], IL + (use ? q : 0), use);
        }
        cp_async4(wil + lane, IL + (bw + lane < s.T ? bw + lane : 0), bw + lane < s.T);
        asm volatile("cp.async.commit_group;\n" ::: "memory");
    }
    // ---- the values this warp reads, every load issued before the first use
    // (their latencies overlap, with each other and with the staging copies):
    // the window band at this thread's fragment entries, and the rung values
    // of the warp's 16 slab columns for all active rungs, rv[i][x] = p or dS of
    // query bw + s0 + x for active rung i in increasing d (0 past the end of
    // the sequence and for the padding entries)
    float bv[NT][4];
#pragma unroll
    for (int j = 0; j < NT; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const bool hi = e >= 2;
            const int r = hi ? g4 + 8 : g4;
            const int x = 8 * j + 2 * c4 + (e & 1);
            const int t = x - r;                              // query - key
            const int q = bw + x;
            const bool use = (hi ? vhi : vlo) && t >= 0 && t <= s.W && q < s.T;
            bv[j][e] = use ? X[(unsigned)(t * s.T + q)] : 0.f;
        }
    float rvv[kMmaMaxRungs * 16 / 32];
#pragma unroll
    for (int j = 0; j < kMmaMaxRungs * 16 / 32; ++j) {
        const int u = lane + 32 * j;
        const int i = u >> 4, x = u & 15;
        const int q = bw + L.act_s0[i] + x;
        const bool use = i < L.n_act && q < s.T;
        rvv[j] = use ? X[(unsigned)((s.W + 1 + L.act_k[i]) * s.T + q)] : 0.f;
    }
    if (IL) {
        asm volatile("cp.async.wait_group 0;\n" ::: "memory");
        __syncwarp();
#pragma unroll
        for (int j = 0; j < NT; ++j)
#pragma unroll
            for (int e = 0; e < 4; ++e) bv[j][e] *= wil[8 * j + 2 * c4 + (e & 1)];
#pragma unroll
        for (int j = 0; j < kMmaMaxRungs * 16 / 32; ++j) {
            const int u = lane + 32 * j;
            rvv[j] *= rv[u >> 4][u & 15];
        }
        __syncwarp();                             // every lane has read its entries before the table is rewritten
    }
#pragma unroll
    for (int j = 0; j < kMmaMaxRungs * 16 / 32; ++j) {
        const int u = lane + 32 * j;
        rv[u >> 4][u & 15] = rvv[j];
    }
    __syncwarp();
    unsigned band[NT][2];
#pragma unroll
    for (int j = 0; j < NT; ++j) {
        band[j][0] = pack_bf16(bv[j][0], bv[j][1]);
        band[j][1] = pack_bf16(bv[j][2], bv[j][3]);
    }
    ok = mbar_wait(bar, parity) && ok;

    const int lv = (lane & 7) + (lane & 8);       // .trans loads: row of the 16-row k-chunk, chunk lane >> 4
    const unsigned avb = row_chunk(sbase, L.win_smem + wrel + lv, lane >> 4);
#pragma unroll
    for (int kk = 0; kk + 1 < NT; kk += 2) {
        const unsigned afr[4] = {band[kk][0], band[kk][1], band[kk + 1][0], band[kk + 1][1]};
#pragma unroll
        for (int n = 0; n < 8; n += 2) {
            unsigned b0, b1, b2, b3;
            ldsm_x4_t((avb ^ (unsigned)(n << 4)) + 1024u * kk, b0, b1, b2, b3);
            mma_bf16_16816(acc[n], afr, b0, b1);
            mma_bf16_16816(acc[n + 1], afr, b2, b3);
        }
    }
    if constexpr (NT & 1) {
        const int kk = NT - 1;
        const unsigned at = row_chunk(sbase, L.win_smem + wrel + 8 * kk + (lane & 7), lane >> 3);
#pragma unroll
        for (int n = 0; n < 8; n += 4) {
            unsigned b0, b1, b2, b3;
            ldsm_x4_t(at ^ (unsigned)(n << 4), b0, b1, b2, b3);
            mma_bf16_1688(acc[n], band[kk][0], band[kk][1], b0);
            mma_bf16_1688(acc[n + 1], band[kk][0], band[kk][1], b1);
            mma_bf16_1688(acc[n + 2], band[kk][0], band[kk][1], b2);
            mma_bf16_1688(acc[n + 3], band[kk][0], band[kk][1], b3);
        }
    }

    // ---- rungs: slab column x is query bw + s0 + x; row r takes x = r (floor
    // side, weight 1-w) and x = r+1 (far side, weight w).  In this thread's A
    // fragment (rows g4, g4+8; columns 2c4, 2c4+1, 2c4+8, 2c4+9) the nonzero
    // pattern depends only on delta = 2c4 - g4: registers a0 (row g4, columns
    // 2c4..) and a3 (row g4+8, columns 2c4+8..) share the coefficients
    //   column x0:   1-w if delta = 0,  w if delta = 1
    //   column x0+1: 1-w if delta = -1, w if delta = 0,
    // a1 (row g4+8, columns 2c4..) is always zero and a2 (row g4, columns
    // 2c4+8..) holds only w at column 8 of row 7 (lane g4 = 7, c4 = 0).
    const int dl = 2 * c4 - g4;
    const float alo = dl == 0 ? 1.f : 0.f, blo = dl == 0 ? -1.f : (dl == 1 ? 1.f : 0.f);
    const float ahi = dl == -1 ? 1.f : 0.f, bhi = dl == -1 ? -1.f : (dl == 0 ? 1.f : 0.f);
    const float m2 = (g4 == 7 && c4 == 0) ? 1.f : 0.f;
    // Rungs whose slab starts before the end of the sequence: a prefix of the
    // list.  Two per iteration (independent work to overlap); an odd count
    // runs one padding entry, whose values are zero.
    int n_use = 0;
    while (n_use < L.n_act && bw + L.act_s0[n_use] < s.T) ++n_use;
#pragma unroll 1
    for (int i = 0; i < n_use; i += 2) {
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int ii = i + u;
            const float w = L.act_w[ii];
            const float clo = fmaf(blo, w, alo), chi = fmaf(bhi, w, ahi);
            const float2 v0 = *reinterpret_cast<const float2*>(&rv[ii][2 * c4]);
            const float2 v8 = *reinterpret_cast<const float2*>(&rv[ii][2 * c4 + 8]);
            const unsigned afr[4] = {pack_bf16(clo * v0.x, chi * v0.y), 0u,
                                     pack_bf16(m2 * w * v8.x, 0.f), pack_bf16(clo * v8.x, chi * v8.y)};
            const unsigned av = row_chunk(sbase, L.act_smem[ii] + wrel + lv, lane >> 4);
#pragma unroll
            for (int n = 0; n < 8; n += 2) {
                unsigned b0, b1, b2, b3;
                ldsm_x4_t(av ^ (unsigned)(n << 4), b0, b1, b2, b3);
                mma_bf16_16816(acc[n], afr, b0, b1);
                mma_bf16_16816(acc[n + 1], afr, b2, b3);
            }
        }
    }
}

// SPLIT: blocks [0, units) take pass 0 (dv) and blocks [units, 2 units) pass
// 1 (dk~) of the same key tiles, for grids too small to fill the GPU with one
// block per tile (grouped-query heads, small batches); else a block runs both
// passes of its tile.
template <int NT, bool SPLIT>
__global__ void __launch_bounds__(kWarps * 32, 2)
bwd_key_mma_kernel(const __grid_constant__ RowMaps tmQ, const __grid_constant__ RowMaps tmG, BwdArgs a,
                   MmaLayout L) {
    // The kernel before this one is the query pass of the same call.  With the
    // forward residuals pass 0 reads only p and dO, which it does not write,
    // so the wait for it comes before pass 1 (dS), whose first block then sums
    // the query pass's rung partials.
    pdl_trigger();
    const int units = (int)a.s.dTiles.d * a.s.B * a.s.Hkv;
    const int pass_first = SPLIT && (int)blockIdx.x >= units ? 1 : 0;
    const int pass_end = SPLIT ? pass_first + 1 : 2;
    const int blk = (int)blockIdx.x - pass_first * units;
    bool waited = a.saved == 0;
    if (waited) pdl_wait();
    extern __shared__ unsigned char smem_raw[];
    __shared__ unsigned long long bar;
    // per warp: rung values of its slab columns; after a pass, its output rows
    __shared__ __align__(16) float rvals[kWarps][kMmaMaxRungs][16];
    __shared__ float wils[kWarps][32];                    // per warp: 1 / row sum of its band queries
    __shared__ float red[kMmaMaxRungs];                   // block 0: dL/dd_k
    __shared__ long long red64[kWarps * kMmaMaxRungs];
    unsigned char* buf = reinterpret_cast<unsigned char*>(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const unsigned sbase = smem_u32(buf);

    const Shape& s = a.s;
    const int bhk = (int)fdiv((unsigned)blk, s.dTiles);   // b * Hkv + hk; blk = bhk * tiles + tile
    const int j0 = (blk - bhk * (int)s.dTiles.d) * kMmaTile;
    const int b = (int)fdiv((unsigned)bhk, s.dHkv), hk = bhk - b * s.Hkv;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g4 = lane >> 2, c4 = lane & 3;
    const int wrel = warp * kRowsPerWarp;
    const int bw = j0 + wrel;
    const int klo = bw + g4, khi = bw + g4 + 8;
    const bool vlo = klo < s.T && g4 < kRowsPerWarp;
    const bool vhi = khi < s.T && g4 + 8 < kRowsPerWarp;

    __shared__ RopeSmem rsm;
    rope_to_smem(rsm, a.rope, L, tid);
    if (tid == 0) {
        mbar_init(&bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    __syncthreads();

    unsigned parity = 0;
    bool ok = true;
    const size_t krow0 = (size_t)bhk * s.T;
#pragma unroll 1
    for (int pass = pass_first; pass < pass_end; ++pass) {  // 0: dv from dO rows; 1: dk~ from q~ rows
        if (pass == 1) {
            if (!waited) pdl_wait();
            waited = true;
            if (blk == 0 && a.want_dd) convert_rung_sums(a, red, red64);
        }
        float acc[8][4];
#pragma unroll
        for (int n = 0; n < 8; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;
#pragma unroll 1
        for (int g = 0; g < s.G; ++g) {
            const int qhead = b * s.H + hk * s.G + g;
            const float* X = (pass ? a.DSs : a.Ps) + (size_t)qhead * a.S * s.T;
            if (warp == 0) {
                const RowMaps& m = pass ? tmQ : tmG;
                issue_rows(buf, &m.m64, &m.m8, L, j0, qhead, &bar, lane);
            }
            if (pass == 0)
                key_pass<NT>(acc, X, a, L, sbase, bw, wrel, g4, c4, lane, vlo, vhi, &bar, parity, ok,
                                 rvals[warp], a.saved ? a.res_il + (size_t)qhead * s.T : nullptr, wils[warp]);
            else
                key_pass<NT>(acc, X, a, L, sbase, bw, wrel, g4, c4, lane, vlo, vhi, &bar, parity, ok,
                                 rvals[warp]);
            parity ^= 1u;
            // every warp is done with the staged rows before the buffer is refilled
            asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
            __syncthreads();
        }
        if (!ok) raise_status(a.status, kStatusWaitTimeout);
        const float sc = ok ? (pass ? s.scale : 1.f) : __int_as_float(0x7fc00000);
        __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(pass ? a.dk : a.dv) + krow0 * kHeadDim;
        // dk = R(-theta key) dk~: cos, sin of pair m = 8n + 2c4 + u (m + 32 in
        // n-tile n + 4) at klo, advanced by 8 positions for khi
        float ec[4][2], es[4][2];
        if (pass) {
#pragma unroll
            for (int n = 0; n < 4; ++n)
#pragma unroll
                for (int u = 0; u < 2; ++u) rope_cs_s(rsm, 8 * n + 2 * c4 + u, klo, ec[n][u], es[n][u]);
        }
        // Rows g4 (half 0) and g4 + 8 (half 1) leave through this warp's table,
        // 8 rows of 128 bytes at a time (16-byte chunk c of row r at chunk
        // c ^ r), and go out as runs of consecutive rows: a warp's stores then
        // cover 512 contiguous bytes instead of 8 rows' 16-byte pieces.
        unsigned* stage = reinterpret_cast<unsigned*>(&rvals[warp][0][0]);
        __syncwarp();                             // the pass's reads of the table are done
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            if (pass && half == 1) {
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
#pragma unroll
            for (int n = 0; n < 8; ++n) {
                acc[n][2 * half] *= sc;
                acc[n][2 * half + 1] *= sc;
            }
            if (pass) {
#pragma unroll
                for (int n = 0; n < 4; ++n) {
#pragma unroll
                    for (int u = 0; u < 2; ++u) {
                        const float xa = acc[n][2 * half + u], xb = acc[n + 4][2 * half + u];
                        acc[n][2 * half + u] = xa * ec[n][u] + xb * es[n][u];
                        acc[n + 4][2 * half + u] = xb * ec[n][u] - xa * es[n][u];
                    }
                }
            }
#pragma unroll
            for (int n = 0; n < 8; ++n)
                stage[g4 * 32 + ((n ^ g4) << 2) + c4] = pack_bf16(acc[n][2 * half], acc[n][2 * half + 1]);
            __syncwarp();
            // rows bw + 8 half + r, r < 8 (7 in the second half: row 15 of the
            // tile is the next warp's), below T
            const int nrow = min(half ? kRowsPerWarp - 8 : 8, s.T - (bw + 8 * half));
#pragma unroll
            for (int c = lane; c < 64; c += 32) {
                const int r = c >> 3, ch = c & 7;
                if (r < nrow) {
                    const uint4 v = *reinterpret_cast<const uint4*>(stage + r * 32 + ((ch ^ r) << 2));
                    *reinterpret_cast<uint4*>(dst + (size_t)(bw + 8 * half + r) * kHeadDim + 8 * ch) = v;
                }
            }
            __syncwarp();                         // the table is read before it is rewritten
        }
    }
}

template <int NT>
cudaError_t launch_nt(const RowMaps& mq, const RowMaps& mg, const BwdArgs& a, const MmaLayout& L,
                      unsigned grid, size_t smem, cudaStream_t st) {
    // one block per tile unless that leaves the GPU under two waves of blocks
    static int slots = 0;
    if (slots == 0) {
        int dev = 0, sms = 0;
        slots = cudaGetDevice(&dev) == cudaSuccess &&
                cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && sms > 0
                    ? 2 * sms : 2 * 152;
    }
    const bool split = (long long)grid < 2LL * slots;
    auto kern = split ? bwd_key_mma_kernel<NT, true> : bwd_key_mma_kernel<NT, false>;
    if (split) grid *= 2;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_kernel(kern, dim3(grid), dim3(kWarps * 32), smem, st, mq, mg, a, L);
}

}  // namespace

size_t bwd_key_mma_static_smem() {
    return sizeof(float) * (kWarps * kMmaMaxRungs * 16 + kWarps * 32 + kMmaMaxRungs) +
           sizeof(long long) * kWarps * kMmaMaxRungs + sizeof(RopeSmem) + 64;
}

size_t bwd_key_mma_smem_bytes(const MmaLayout& L, bool) { return fwd_mma_smem_bytes(L); }

int bwd_key_mma_blocks(const Shape& s) {
    const long long tiles = (s.T + kMmaTile - 1) / kMmaTile;
    return (int)(tiles * s.B * s.Hkv);
}

cudaError_t launch_bwd_key_mma(const BwdArgs& a, const MmaLayout& L, cudaStream_t st) {
    const long long grid = bwd_key_mma_blocks(a.s);
    if (grid <= 0) return cudaSuccess;
    RowMaps mq, mg;
    const int heads = a.s.B * a.s.H;
    if (!encode_row_maps(&mq, a.qt, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.s.T, heads) ||
        !encode_row_maps(&mg, a.dout, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a.s.T, heads))
        return cudaErrorInvalidValue;
    const size_t smem = bwd_key_mma_smem_bytes(L, a.saved != 0);
    switch (L.nt) {
    case 2: return launch_nt<2>(mq, mg, a, L, (unsigned)grid, smem, st);
    case 3: return launch_nt<3>(mq, mg, a, L, (unsigned)grid, smem, st);
    default: return launch_nt<4>(mq, mg, a, L, (unsigned)grid, smem, st);
    }
}

}  // namespace fibattn
