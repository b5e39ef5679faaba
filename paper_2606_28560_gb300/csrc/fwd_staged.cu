// fwd_staged.cu -- forward pass with shared-memory staging and register
// blocking (arXiv 2606.28560, Section 2 "Attended set").
//
// Rung offsets are shared by every query (Section 2), so for a tile of M
// consecutive queries each slot group reads a contiguous shifted slab of key
// rows: the window band [i0-W, i0+M) and, per rung, [i0-s0-1, i0+M-s0).  The
// host merges these intervals once per launch; each CTA copies the union of
// its rows into shared memory once (cp.async, rows outside [0, T) zero-filled),
// first the RoPE-rotated keys, then -- into the same buffer -- the values.
//
// Thread layout: a warp holds 4 groups of 8 lanes; lane (g, c) owns head dims
// 8c..8c+7 of the R consecutive queries of group g.  A row chunk loaded once
// serves every query of the group that reads that row: a rung slab of R+1
// rows feeds 2R (query, row) pairs; the window band of R+W rows feeds R(W+1).
// Partial dot products over 8 dims are combined across the 8 lanes by a
// transposed butterfly, after which lane c holds whole scores.
//
//   phase 1: scores (window + interpolated rungs) -> shared scores [M][S]
//   phase 2: per-query softmax (one thread per query) -> probabilities, lse
//   phase 3: probability-weighted values (equally interpolated rungs) -> O
#include "fibattn_internal.cuh"
#include "fwd_staged.cuh"

namespace fibattn {
namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem, bool full) {
    unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    int src_size = full ? 16 : 0;                // 0: write 16 zero bytes, read nothing
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" :: "r"(s), "l"(gmem), "r"(src_size));
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;\n" ::); }

// Copy the union of the tile's rows (128 B each) into shared memory.
__device__ __forceinline__ void stage_rows(char* rows_sm, const char* head, const StageLayout& L, int i0, int T) {
    const int tid = threadIdx.x, nt = blockDim.x;
    for (int iv = 0; iv < L.n_iv; ++iv) {
        const int start = i0 + L.iv_start[iv], len = L.iv_len[iv], sm0 = L.iv_smem[iv];
        for (int idx = tid; idx < len * 8; idx += nt) {
            const int row = idx >> 3, ch = idx & 7;
            const int abs_row = start + row;
            const bool ok = abs_row >= 0 && abs_row < T;
            const char* src = head + ((size_t)(ok ? abs_row : 0) * 128 + ch * 16);
            cp_async16(rows_sm + ((size_t)(sm0 + row) * 128 + ch * 16), src, ok);
        }
    }
}

// 8 consecutive elements of a staged row (16 B) as fp32.
__device__ __forceinline__ void lds8(const char* p, const __half*, float* x) {
    uint4 u = *reinterpret_cast<const uint4*>(p);
    unsigned w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float2 f = __half22float2(*reinterpret_cast<__half2*>(&w[i]));
        x[2 * i] = f.x; x[2 * i + 1] = f.y;
    }
}
__device__ __forceinline__ void lds8(const char* p, const __nv_bfloat16*, float* x) {
    uint4 u = *reinterpret_cast<const uint4*>(p);
    unsigned w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        x[2 * i] = __uint_as_float(w[i] << 16);
        x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}

__device__ __forceinline__ float dot8(const float* a, const float* b) {
    float s = a[0] * b[0];
#pragma unroll
    for (int e = 1; e < 8; ++e) s = fmaf(a[e], b[e], s);
    return s;
}

// Transposed butterfly over the 8 lanes c = lane & 7 of a group: on entry
// v[r] is this lane's partial (8 dims) for query r (r < R); on exit the
// return value is the full score of query r = c >> log2(8/R) (lanes sharing
// a query hold the same value).
template <int R>
__device__ __forceinline__ float group_transpose_sum(float* v, int lane) {
    if constexpr (R == 8) {
        const bool b2 = lane & 4, b1 = lane & 2, b0 = lane & 1;
        float w4[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            float send = b2 ? v[j] : v[j + 4];
            float keep = b2 ? v[j + 4] : v[j];
            w4[j] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
        }
        float w2[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            float send = b1 ? w4[j] : w4[j + 2];
            float keep = b1 ? w4[j + 2] : w4[j];
            w2[j] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
        }
        float send = b0 ? w2[0] : w2[1];
        float keep = b0 ? w2[1] : w2[0];
        return keep + __shfl_xor_sync(0xffffffffu, send, 1);
    } else {  // R == 4
        const bool b2 = lane & 4, b1 = lane & 2;
        float w2[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            float send = b2 ? v[j] : v[j + 2];
            float keep = b2 ? v[j + 2] : v[j];
            w2[j] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
        }
        float send = b1 ? w2[0] : w2[1];
        float keep = b1 ? w2[1] : w2[0];
        float x = keep + __shfl_xor_sync(0xffffffffu, send, 2);
        return x + __shfl_xor_sync(0xffffffffu, x, 1);
    }
}

template <typename T, int R>
__global__ void __launch_bounds__(8 * kStagedM / R) fwd_staged_kernel(FwdArgs a, StageLayout L) {
    grid_dependency_sync();
    using RT = typename RotOf<T>::type;
    constexpr int M = kStagedM;
    constexpr int QPW = 4 * R;                   // queries per warp
    extern __shared__ __align__(16) char smem[];
    char* rows_sm = smem;
    float* S_sm = reinterpret_cast<float*>(smem + (size_t)L.rows * 128);   // [M][SP]

    const Shape s = a.s;
    const int SP = L.slot_pitch;
    const int nslot = s.W + 1 + a.r.K;
    const int tiles = (s.T + M - 1) / M;
    const int bh = blockIdx.x / tiles;
    const int i0 = (blockIdx.x % tiles) * M;
    const int b = bh / s.H, h = bh % s.H, hk = h / s.G;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int g = lane >> 3, c = lane & 7;
    const int qw = warp * QPW + g * R;           // tile-relative first query of the group
    const int u0 = i0 + qw;                      // absolute first query of the group
    constexpr int kShift = (R == 8) ? 0 : 1;     // query of lane c after the butterfly: c >> kShift
    const int myq = qw + (c >> kShift);          // tile-relative query whose score this lane holds
    const int myi = i0 + myq;

    const char* khead = reinterpret_cast<const char*>(reinterpret_cast<const RT*>(a.kt) +
                                                      ((size_t)(b * s.Hkv + hk) * s.T) * kHeadDim);
    const char* vhead = reinterpret_cast<const char*>(reinterpret_cast<const T*>(a.v) +
                                                      ((size_t)(b * s.Hkv + hk) * s.T) * kHeadDim);

    // ---- stage rotated keys; meanwhile mark every score slot as unattended
    stage_rows(rows_sm, khead, L, i0, s.T);
    asm volatile("cp.async.commit_group;\n" ::);
    for (int idx = tid; idx < M * SP; idx += blockDim.x) S_sm[idx] = -INFINITY;

    // ---- q~ for the R queries of this group, dims 8c..8c+7 (RoPE pairs m, m+32)
    float qf[R][8];
    {
        const T* Q = reinterpret_cast<const T*>(a.q) + ((size_t)bh * s.T) * kHeadDim;
        const int cc = c & 3;                     // pair block: m = 8cc + e
        const bool hi = c >= 4;                   // this lane holds the second halves
        float cs[8], sn[8], c1[8], s1[8];
        const int p0 = min(u0, s.T - 1);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            rope_cs(a.rope, 8 * cc + e, p0, cs[e], sn[e]);
            c1[e] = L.rope_c1[8 * cc + e];
            s1[e] = L.rope_s1[8 * cc + e];
        }
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int i = min(u0 + r, s.T - 1);
            float own[8], oth[8];
            Vec8<T>::load(Q + (size_t)i * kHeadDim + 8 * c, own);
            Vec8<T>::load(Q + (size_t)i * kHeadDim + 8 * (c ^ 4), oth);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                // R(pos): x' = x c - y s, y' = y c + x s for the pair (x, y) = (first, second)
                qf[r][e] = hi ? (own[e] * cs[e] + oth[e] * sn[e]) : (own[e] * cs[e] - oth[e] * sn[e]);
            }
            if (r + 1 < R) {
#pragma unroll
                for (int e = 0; e < 8; ++e) {      // advance the angle by one position
                    const float cn = cs[e] * c1[e] - sn[e] * s1[e];
                    const float sn2 = sn[e] * c1[e] + cs[e] * s1[e];
                    cs[e] = cn; sn[e] = sn2;
                }
            }
        }
    }
    const float sc2 = s.scale * kLog2e;           // scores kept in log2 units

    cp_async_wait_all();
    __syncthreads();

    // ---- phase 1a: window band.  Row u0+rel serves query r at slot t = r - rel.
    float part[R];
    for (int rel = -s.W; rel < R; ++rel) {
        float kr[8];
        lds8(rows_sm + (size_t)(L.win_smem + qw + rel) * 128 + c * 16, (const RT*)nullptr, kr);
#pragma unroll
        for (int r = 0; r < R; ++r) part[r] = dot8(qf[r], kr);
        const float sco = group_transpose_sum<R>(part, lane);
        const int t = (myq - qw) - rel;
        if (t >= 0 && t <= s.W && myi - t >= 0 && myi < s.T && ((c & ((1 << kShift) - 1)) == 0))
            S_sm[myq * SP + t] = sco * sc2;
    }
    // ---- phase 1b: rungs.  Slab row x (absolute u0-s0-1+x) is the far row of
    // query x (weight w) and the floor row of query x-1 (weight 1-w).
    for (int k = 0; k < a.r.K; ++k) {
        if (!((a.r.active >> k) & 1u)) continue;
        if (a.r.d[k] > (float)(i0 + M - 1)) continue;         // masked for the whole tile
        const float w = a.r.w[k], w1 = 1.f - w;
        const char* slab = rows_sm + (size_t)(L.rung_smem[k] + qw) * 128 + c * 16;
#pragma unroll
        for (int r = 0; r < R; ++r) part[r] = 0.f;
        if (w != 0.f) {
#pragma unroll
            for (int x = 0; x <= R; ++x) {
                float kr[8];
                lds8(slab + x * 128, (const RT*)nullptr, kr);
                if (x < R) part[x] = fmaf(w, dot8(qf[x], kr), part[x]);
                if (x >= 1) part[x - 1] = fmaf(w1, dot8(qf[x - 1], kr), part[x - 1]);
            }
        } else {
#pragma unroll
            for (int x = 1; x <= R; ++x) {
                float kr[8];
                lds8(slab + x * 128, (const RT*)nullptr, kr);
                part[x - 1] = dot8(qf[x - 1], kr);
            }
        }
        const float sco = group_transpose_sum<R>(part, lane);
        if (a.r.d[k] <= (float)myi && myi < s.T && ((c & ((1 << kShift) - 1)) == 0))
            S_sm[myq * SP + s.W + 1 + k] = sco * sc2;
    }
    __syncthreads();

    // ---- stage values into the same buffer (all key reads are done)
    stage_rows(rows_sm, vhead, L, i0, s.T);
    asm volatile("cp.async.commit_group;\n" ::);

    // ---- phase 2: softmax, one thread per query (scores in log2 units)
    if (tid < M) {
        float* row = S_sm + tid * SP;
        float m = -INFINITY;
        for (int j = 0; j < nslot; ++j) m = fmaxf(m, row[j]);
        float l = 0.f;
        for (int j = 0; j < nslot; ++j) {
            const float p = exp2f(row[j] - m);   // unattended slots: exp2(-inf) = 0
            row[j] = p;
            l += p;
        }
        const float inv = 1.f / l;
        for (int j = 0; j < nslot; ++j) row[j] *= inv;
        const int i = i0 + tid;
        if (i < s.T) a.lse[(size_t)bh * s.T + i] = (m + __log2f(l)) * kLn2;
    }
    cp_async_wait_all();
    __syncthreads();

    // ---- phase 3a: window band of values
    float acc[R][8];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[r][e] = 0.f;
    for (int rel = -s.W; rel < R; ++rel) {
        float vr[8];
        lds8(rows_sm + (size_t)(L.win_smem + qw + rel) * 128 + c * 16, (const T*)nullptr, vr);
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int t = r - rel;
            if (t >= 0 && t <= s.W) {
                const float p = S_sm[(qw + r) * SP + t];
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[r][e] = fmaf(p, vr[e], acc[r][e]);
            }
        }
    }
    // ---- phase 3b: rungs, values interpolated with the same weights
    for (int k = 0; k < a.r.K; ++k) {
        if (!((a.r.active >> k) & 1u)) continue;
        if (a.r.d[k] > (float)(i0 + M - 1)) continue;
        const float w = a.r.w[k], w1 = 1.f - w;
        const char* slab = rows_sm + (size_t)(L.rung_smem[k] + qw) * 128 + c * 16;
        float p[R];
#pragma unroll
        for (int r = 0; r < R; ++r) p[r] = S_sm[(qw + r) * SP + s.W + 1 + k];
#pragma unroll
        for (int x = 0; x <= R; ++x) {
            if (x == 0 && w == 0.f) continue;     // integer rung: no far row
            float vr[8];
            lds8(slab + x * 128, (const T*)nullptr, vr);
            if (x < R) {
                const float pw = p[x] * w;
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[x][e] = fmaf(pw, vr[e], acc[x][e]);
            }
            if (x >= 1) {
                const float pw = p[x - 1] * w1;
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[x - 1][e] = fmaf(pw, vr[e], acc[x - 1][e]);
            }
        }
    }
    // ---- store O: the 8 lanes of a group write one 128 B row per query
    T* O = reinterpret_cast<T*>(a.out) + ((size_t)bh * s.T) * kHeadDim;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int i = u0 + r;
        if (i < s.T) Vec8<T>::store(O + (size_t)i * kHeadDim + 8 * c, acc[r]);
    }
}

}  // namespace

size_t fwd_staged_smem_bytes(const StageLayout& L) {
    return (size_t)L.rows * 128 + (size_t)kStagedM * L.slot_pitch * 4;
}

cudaError_t launch_fwd_staged(const FwdArgs& a, const StageLayout& L, bool bf16, cudaStream_t st) {
    const long long tiles = (a.s.T + kStagedM - 1) / kStagedM;
    const long long grid = tiles * a.s.B * a.s.H;
    if (grid <= 0) return cudaSuccess;
    const size_t smem = fwd_staged_smem_bytes(L);
    constexpr int R = kStagedR;
    constexpr int threads = 8 * kStagedM / R;
    if (!bf16) return cudaErrorInvalidValue;     // fp32 I/O uses the row-gather kernel
    auto kern = fwd_staged_kernel<__nv_bfloat16, R>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_kernel(kern, dim3((unsigned)grid), dim3(threads), smem, st, a, L);
}

}  // namespace fibattn
