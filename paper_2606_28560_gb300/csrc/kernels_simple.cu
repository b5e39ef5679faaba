// kernels_simple.cu -- straightforward CUDA kernels for every step of the
// path (arXiv 2606.28560, Section 2): the RoPE prologue, the forward pass and
// the backward pass.  Rows are read through L1/L2 with 128-bit loads; a group
// of 4 lanes owns one query (or key) row, each lane 8 RoPE pairs (16 dims).
//
// Forward  (Section 2, "Attended set"): online softmax over the window slots
//          t = 0..W and the interpolated rungs, accumulating the equally
//          interpolated values.
// Backward (chain rule of the forward): a query-centric pass recomputes the
//          probabilities, forms dL/dscore, dq and the per-rung distance
//          gradient; a key-centric pass gathers dk and dv from the shifted
//          query rows (no atomics); a one-block pass sums the per-block rung
//          partials in a fixed order and applies d_k = alpha f_k and
//          alpha = 0.5 + sigmoid(theta) (Section 2, "The per-layer scalar").
#include <algorithm>

#include "fibattn_internal.cuh"

namespace fibattn {

namespace {

constexpr int kThreads = 128;                 // 4 warps
constexpr int kRowsPerBlock = kThreads / 4;   // 32 query/key rows per block
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ float group_sum(float x) {
    x += __shfl_xor_sync(0xffffffffu, x, 1);
    x += __shfl_xor_sync(0xffffffffu, x, 2);
    return x;
}

// Packed fp32 pairs: one fma.rn.f32x2 issue performs two FMAs.
template <typename T>
__device__ __forceinline__ void load_chunk2(const T* row, int c, float2* x) {
    float t[16];
    load_chunk(row, c, t);
#pragma unroll
    for (int i = 0; i < 8; ++i) x[i] = make_float2(t[2 * i], t[2 * i + 1]);
}
__device__ __forceinline__ float dot16x2(const float2* a, const float2* b) {
    float2 acc = __fmul2_rn(a[0], b[0]);
#pragma unroll
    for (int i = 1; i < 8; ++i) acc = __ffma2_rn(a[i], b[i], acc);
    return acc.x + acc.y;
}
__device__ __forceinline__ void axpy16x2(float a, const float2* x, float2* y) {
    const float2 a2 = make_float2(a, a);
#pragma unroll
    for (int i = 0; i < 8; ++i) y[i] = __ffma2_rn(a2, x[i], y[i]);
}

// ---------------------------------------------------------------- RoPE ----

template <typename T, typename R>
__global__ void __launch_bounds__(256) rope_rows_kernel(const T* __restrict__ src, R* __restrict__ dst,
                                                        long long rows, int T_, RopeParams rp) {
    grid_dependency_sync();
    // One (row, 8-pair chunk) item per thread per pass; grid-stride over items.
    const long long n = rows * 4;
    for (long long g = blockIdx.x * (long long)blockDim.x + threadIdx.x; g < n;
         g += (long long)gridDim.x * blockDim.x) {
        const long long row = g >> 2;
        const int c = (int)(g & 3);
        float x[16];
        load_chunk(src + row * kHeadDim, c, x);
        rope_chunk(rp, (int)(row % T_), c, x, false);
        store_chunk(dst + row * kHeadDim, c, x);
    }
}

// bf16 rows in, fp16 rotated rows out.  A block tile is kRopePos consecutive
// positions of TH heads: the tile's cos/sin (one pair and position per
// thread, evaluated before the wait for the previous kernel) go to shared
// memory, and every row of the tile reads them from there, so an angle is
// evaluated once per tile instead of once per head.  Thread item = (head,
// position, chunk c): dims 8c..8c+7 and their RoPE partners 32+8c..32+8c+7;
// a warp covers the tile's 8 positions x 4 chunks of one head (1 KB
// contiguous), and a thread issues the loads of all its items (TH / 8)
// before any arithmetic.
constexpr int kRopePos = 8;
constexpr int kRopeTabStride = 34;            // floats per position (32 + pad: conflict-free float2 reads)
template <int TH>
__global__ void __launch_bounds__(256) rope_rows_bf16_kernel(const __nv_bfloat16* __restrict__ src,
                                                             __half* __restrict__ dst, int heads, int T_,
                                                             RopeParams rp, unsigned* status) {
    constexpr int kItems = TH / 8;                // per thread (256 threads)
    __shared__ __align__(16) float ctab[kRopePos * kRopeTabStride], stab[kRopePos * kRopeTabStride];
    const int tid = threadIdx.x;
    const int c = tid & 3, pr = (tid >> 2) & 7, hr0 = tid >> 5;
    const int tiles_p = (T_ + kRopePos - 1) / kRopePos;
    const long long tiles = (long long)tiles_p * ((heads + TH - 1) / TH);
    float rmax = 0.f;                             // largest |rotated entry|: fp16 holds < 65520
    bool waited = false;
    for (long long tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
        const int tp = (int)(tile % tiles_p), th = (int)(tile / tiles_p);
        const int p0 = tp * kRopePos, h0 = th * TH;
        {                                         // pair m = tid & 31 at position p0 + (tid >> 5)
            float cs, sn;
            rope_cs(rp, tid & 31, p0 + (tid >> 5), cs, sn);
            ctab[(tid >> 5) * kRopeTabStride + (tid & 31)] = cs;
            stab[(tid >> 5) * kRopeTabStride + (tid & 31)] = sn;
        }
        if (!waited) {
            grid_dependency_sync();
            waited = true;
        }
        const int p = p0 + pr;
        uint4 raw[kItems][2];
#pragma unroll
        for (int u = 0; u < kItems; ++u) {
            const int h = h0 + hr0 + 8 * u;
            if (h < heads && p < T_) {
                const __nv_bfloat16* row = src + ((size_t)h * T_ + p) * kHeadDim;
                raw[u][0] = *reinterpret_cast<const uint4*>(row + 8 * c);
                raw[u][1] = *reinterpret_cast<const uint4*>(row + kHalf + 8 * c);
            }
        }
        __syncthreads();                          // the tile's cos/sin are in shared memory
        const float2* cp = reinterpret_cast<const float2*>(ctab + pr * kRopeTabStride + 8 * c);
        const float2* sp = reinterpret_cast<const float2*>(stab + pr * kRopeTabStride + 8 * c);
#pragma unroll
        for (int u = 0; u < kItems; ++u) {
            const int h = h0 + hr0 + 8 * u;
            if (h >= heads || p >= T_) continue;
            const unsigned* wa = reinterpret_cast<const unsigned*>(&raw[u][0]);
            const unsigned* wb = reinterpret_cast<const unsigned*>(&raw[u][1]);
            unsigned oa[4], ob[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float a0 = __uint_as_float(wa[e] << 16), a1 = __uint_as_float(wa[e] & 0xffff0000u);
                const float b0 = __uint_as_float(wb[e] << 16), b1 = __uint_as_float(wb[e] & 0xffff0000u);
                const float2 ce = cp[e], se = sp[e];         // pairs (8c + 2e, 32 + 8c + 2e) and the next
                const float xa0 = a0 * ce.x - b0 * se.x, xa1 = a1 * ce.y - b1 * se.y;
                const float xb0 = b0 * ce.x + a0 * se.x, xb1 = b1 * ce.y + a1 * se.y;
                rmax = fmaxf(rmax, fmaxf(fmaxf(fabsf(xa0), fabsf(xa1)), fmaxf(fabsf(xb0), fabsf(xb1))));
                __half2 ra = __floats2half2_rn(xa0, xa1);
                __half2 rb = __floats2half2_rn(xb0, xb1);
                oa[e] = *reinterpret_cast<unsigned*>(&ra);
                ob[e] = *reinterpret_cast<unsigned*>(&rb);
            }
            __half* row = dst + ((size_t)h * T_ + p) * kHeadDim;
            *reinterpret_cast<uint4*>(row + 8 * c) = make_uint4(oa[0], oa[1], oa[2], oa[3]);
            *reinterpret_cast<uint4*>(row + kHalf + 8 * c) = make_uint4(ob[0], ob[1], ob[2], ob[3]);
        }
        __syncthreads();                          // read before the next tile rewrites them
    }
    if (!waited) grid_dependency_sync();
    if (rmax >= 65520.f) raise_status(status, kStatusRange);
}

// ------------------------------------------------------------- forward ----

template <typename T>
__global__ void __launch_bounds__(kThreads) fwd_simple_kernel(FwdArgs a) {
    grid_dependency_sync();
    const Shape s = a.s;
    const int lane = threadIdx.x & 31, c = lane & 3;
    const int tiles = (s.T + kRowsPerBlock - 1) / kRowsPerBlock;
    const int bh = blockIdx.x / tiles;
    const int i = (blockIdx.x % tiles) * kRowsPerBlock + (threadIdx.x >> 2);
    const int b = bh / s.H, h = bh % s.H, hk = h / s.G;
    const bool qvalid = i < s.T;
    const int ii = qvalid ? i : s.T - 1;

    const T* Q = reinterpret_cast<const T*>(a.q) + ((size_t)bh * s.T) * kHeadDim;
    using R = typename RotOf<T>::type;
    const R* Kt = reinterpret_cast<const R*>(a.kt) + ((size_t)(b * s.Hkv + hk) * s.T) * kHeadDim;
    const T* V = reinterpret_cast<const T*>(a.v) + ((size_t)(b * s.Hkv + hk) * s.T) * kHeadDim;

    float2 q[8];
    {
        float qs[16];
        load_chunk(Q + (size_t)ii * kHeadDim, c, qs);
        rope_chunk(a.rope, ii, c, qs, false);
#pragma unroll
        for (int e = 0; e < 8; ++e) q[e] = make_float2(qs[2 * e], qs[2 * e + 1]);
    }
    const float sc2 = s.scale * kLog2e;          // scores kept in log2 units

    // Scores use the same pairwise dot product as the backward recompute, so
    // both sides round a score identically.
    float m = -INFINITY, l = 0.f;
    float2 acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = make_float2(0.f, 0.f);

    float2 kr[8], vr[8];
    // window slots: distance t = 0..W (self always present)
    for (int t = 0; t <= s.W; ++t) {
        const int j = ii - t;
        const bool ok = j >= 0;
        const int jj = ok ? j : 0;
        load_chunk2(Kt + (size_t)jj * kHeadDim, c, kr);
        const float sco = group_sum(dot16x2(q, kr)) * sc2;
        if (ok) {
            load_chunk2(V + (size_t)jj * kHeadDim, c, vr);
            if (sco > m) {
                const float corr = exp2f(m - sco);
                l *= corr;
                const float2 c2 = make_float2(corr, corr);
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[e] = __fmul2_rn(acc[e], c2);
                m = sco;
            }
            const float p = exp2f(sco - m);
            l += p;
            axpy16x2(p, vr, acc);
        }
        if (__all_sync(0xffffffffu, !ok)) break;
    }
    // rungs: d_k = alpha f_k, read between rows i-s0 (weight 1-w) and i-s0-1 (weight w)
    const float fi = (float)ii;
    for (int k = 0; k < a.r.K; ++k) {
        if (!((a.r.active >> k) & 1u)) continue;
        const int s0 = a.r.s0[k];
        const float w = a.r.w[k];
        const bool ok = a.r.d[k] <= fi;
        const int j0 = ii - s0, j1 = j0 - 1;
        const int jj0 = ok ? j0 : 0;
        load_chunk2(Kt + (size_t)jj0 * kHeadDim, c, kr);
        float sraw = (1.f - w) * dot16x2(q, kr);
        const bool far = w != 0.f;               // warp-uniform
        float2 kf[8];
        if (far) {
            const int jj1 = (ok && j1 >= 0) ? j1 : 0;
            load_chunk2(Kt + (size_t)jj1 * kHeadDim, c, kf);
            if (ok && j1 >= 0) sraw = fmaf(w, dot16x2(q, kf), sraw);
        }
        const float sco = group_sum(sraw) * sc2;
        if (ok) {
            load_chunk2(V + (size_t)jj0 * kHeadDim, c, vr);
            if (sco > m) {
                const float corr = exp2f(m - sco);
                l *= corr;
                const float2 c2 = make_float2(corr, corr);
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[e] = __fmul2_rn(acc[e], c2);
                m = sco;
            }
            const float p = exp2f(sco - m);
            l += p;
            axpy16x2(p * (1.f - w), vr, acc);
            if (far && j1 >= 0) {
                load_chunk2(V + (size_t)j1 * kHeadDim, c, vr);
                axpy16x2(p * w, vr, acc);
            }
        }
    }
    if (qvalid) {
        const float inv = 1.f / l;
        float o[16];
#pragma unroll
        for (int e = 0; e < 8; ++e) { o[2 * e] = acc[e].x * inv; o[2 * e + 1] = acc[e].y * inv; }
        T* O = reinterpret_cast<T*>(a.out) + ((size_t)bh * s.T + i) * kHeadDim;
        store_chunk(O, c, o);
        if (c == 0) a.lse[(size_t)bh * s.T + i] = (m + __log2f(l)) * kLn2;
    }
}

// ------------------------------------------------------------ backward ----

// Query-centric pass, one sweep over the attended slots of query i.  With
// p = exp(score - lse), dp = dO . val and Delta = sum_slots p dp (= dO . o),
// dL/dscore = p (dp - Delta), so
//   dq~ = scale sum_slots p (dp - Delta) key = scale (A - Delta B),
//   A = sum p dp key,  B = sum p key,
// and for rung k (d key / d d_k = k~[j1] - k~[j0], d val / d d_k = v[j1] - v[j0];
// row -1 is a zero row)
//   dL/dd_k += scale p (dp - Delta) q~.(k~[j1]-k~[j0]) + p dO.(v[j1]-v[j0])
//            = t1 - Delta t2,  t1 = scale p ds_k dp + p ddp_k,  t2 = scale p ds_k.
// A, B, t1, t2 and Delta accumulate in the same sweep.  P, dp (per slot, zero
// where not attended) and Delta (per query) go to the workspace for the key
// pass, which forms dL/dscore = P (dp - Delta).
template <typename T>
__global__ void __launch_bounds__(kThreads) bwd_query_kernel(BwdArgs a) {
    grid_dependency_sync();
    __shared__ float tsm[kRowsPerBlock][kMaxRungs][2];   // per-query t1, t2 of each rung
    __shared__ float dsm[kRowsPerBlock];                 // per-query Delta (0 when i >= T)
    const Shape s = a.s;
    const int lane = threadIdx.x & 31, c = lane & 3, warp = threadIdx.x >> 5;
    const int tiles = (s.T + kRowsPerBlock - 1) / kRowsPerBlock;
    const int bh = blockIdx.x / tiles;
    const int i = (blockIdx.x % tiles) * kRowsPerBlock + (threadIdx.x >> 2);
    const int b = bh / s.H, h = bh % s.H, hk = h / s.G;
    const bool qvalid = i < s.T;
    const int ii = qvalid ? i : s.T - 1;
    const float fi = (float)ii;
    const float lse2 = qvalid ? a.lse[(size_t)bh * s.T + ii] * kLog2e : 0.f;
    const float sc2 = s.scale * kLog2e;

    using R = typename RotOf<T>::type;
    const R* Qt = reinterpret_cast<const R*>(a.qt) + ((size_t)bh * s.T) * kHeadDim;
    const T* dO = reinterpret_cast<const T*>(a.dout) + ((size_t)bh * s.T) * kHeadDim;
    const R* Kt = reinterpret_cast<const R*>(a.kt) + ((size_t)(b * s.Hkv + hk) * s.T) * kHeadDim;
    const T* V = reinterpret_cast<const T*>(a.v) + ((size_t)(b * s.Hkv + hk) * s.T) * kHeadDim;
    float* Prow = a.P + ((size_t)bh * s.T + ii) * a.S;
    float* DProw = a.DP + ((size_t)bh * s.T + ii) * a.S;

    float2 q[8], go[8], kr[8], kf[8], vr[8], vf[8];
    load_chunk2(Qt + (size_t)ii * kHeadDim, c, q);
    load_chunk2(dO + (size_t)ii * kHeadDim, c, go);

    float2 A[8], Bv[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) { A[e] = make_float2(0.f, 0.f); Bv[e] = make_float2(0.f, 0.f); }
    float delta = 0.f;
    const int qloc = threadIdx.x >> 2;
    if (c == 0)
        for (int k = 0; k < kMaxRungs; ++k) { tsm[qloc][k][0] = 0.f; tsm[qloc][k][1] = 0.f; }

    // window slots t = 0..W
    for (int t = 0; t <= s.W; ++t) {
        const int j = ii - t;
        const bool ok = j >= 0;
        const int jj = ok ? j : 0;
        load_chunk2(Kt + (size_t)jj * kHeadDim, c, kr);
        load_chunk2(V + (size_t)jj * kHeadDim, c, vr);
        const float sco = group_sum(dot16x2(q, kr)) * sc2;
        const float dp = group_sum(dot16x2(go, vr));
        const float p = ok ? exp2f(sco - lse2) : 0.f;
        const float pdp = p * dp;
        delta += pdp;
        axpy16x2(pdp, kr, A);
        axpy16x2(p, kr, Bv);
        if (qvalid && c == 0) { Prow[t] = p; DProw[t] = ok ? dp : 0.f; }
        if (__all_sync(0xffffffffu, j < 0)) {
            if (qvalid && c == 0)
                for (int u = t + 1; u <= s.W; ++u) { Prow[u] = 0.f; DProw[u] = 0.f; }
            break;
        }
    }
    // rungs
    for (int k = 0; k < a.r.K; ++k) {
        const int slot = s.W + 1 + k;
        if (!((a.r.active >> k) & 1u)) {
            if (qvalid && c == 0) { Prow[slot] = 0.f; DProw[slot] = 0.f; }
            continue;
        }
        const int s0 = a.r.s0[k];
        const float w = a.r.w[k];
        const bool ok = a.r.d[k] <= fi;
        const int j0 = ok ? ii - s0 : 0;
        const bool hasf = ok && j0 >= 1;          // far row -1 is a zero row
        const int j1 = hasf ? j0 - 1 : 0;
        load_chunk2(Kt + (size_t)j0 * kHeadDim, c, kr);
        load_chunk2(V + (size_t)j0 * kHeadDim, c, vr);
        load_chunk2(Kt + (size_t)j1 * kHeadDim, c, kf);
        load_chunk2(V + (size_t)j1 * kHeadDim, c, vf);
        float s0r = dot16x2(q, kr), dp0 = dot16x2(go, vr), s1r = 0.f, dp1 = 0.f;
        if (hasf) { s1r = dot16x2(q, kf); dp1 = dot16x2(go, vf); }
        s0r = group_sum(s0r); s1r = group_sum(s1r);
        dp0 = group_sum(dp0); dp1 = group_sum(dp1);
        const float w1 = 1.f - w;
        const float sco = (w1 * s0r + w * s1r) * sc2;
        const float dp = w1 * dp0 + w * dp1;
        const float p = ok ? exp2f(sco - lse2) : 0.f;
        const float pdp = p * dp;
        delta += pdp;
        const float fw1 = hasf ? w : 0.f;
        axpy16x2(pdp * w1, kr, A);
        axpy16x2(pdp * fw1, kf, A);
        axpy16x2(p * w1, kr, Bv);
        axpy16x2(p * fw1, kf, Bv);
        const float psd = s.scale * p * (s1r - s0r);
        if (c == 0) { tsm[qloc][k][0] = psd * dp + p * (dp1 - dp0); tsm[qloc][k][1] = psd; }
        if (qvalid && c == 0) { Prow[slot] = p; DProw[slot] = ok ? dp : 0.f; }
    }
    if (qvalid) {
        float dq[16];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            dq[2 * e] = s.scale * (A[e].x - delta * Bv[e].x);
            dq[2 * e + 1] = s.scale * (A[e].y - delta * Bv[e].y);
        }
        rope_chunk(a.rope, ii, c, dq, true);
        T* dQ = reinterpret_cast<T*>(a.dq) + ((size_t)bh * s.T + i) * kHeadDim;
        store_chunk(dQ, c, dq);
        if (c == 0) a.Delta[(size_t)bh * s.T + i] = delta;
    }
    if (c == 0) dsm[qloc] = qvalid ? delta : 0.f;
    __syncthreads();
    // per-block rung partials sum_i (t1 - Delta_i t2), queries in a fixed order
    float x = 0.f;
    if (threadIdx.x < a.r.K) {
        const int k = threadIdx.x;
        for (int u = 0; u < kRowsPerBlock; ++u) {
            const bool valid = (blockIdx.x % tiles) * kRowsPerBlock + u < s.T;
            if (valid) x += tsm[u][k][0] - dsm[u] * tsm[u][k][1];
        }
    }
    if (a.want_dd) write_rung_partials(a, x);
}

// Key-centric pass.  Key row j of kv head hk receives, from every query head
// of its group, the slots that read it: window slot t of query j+t (weight 1),
// rung k of query j+s0_k (floor row, weight 1-w_k) and of query j+s0_k+1 (far
// row, weight w_k):  dk~_j = scale sum c dS q~_i,  dv_j = sum c P dO_i, with
// dS = P (dp - Delta_i) from the query pass.
template <typename T>
__global__ void __launch_bounds__(kThreads) bwd_key_kernel(BwdArgs a) {
    grid_dependency_sync();
    __shared__ float red[kMaxRungs];
    __shared__ long long red64[(kThreads / 32) * kMaxRungs];
    if (blockIdx.x == 0 && a.want_dd) convert_rung_sums(a, red, red64);
    const Shape s = a.s;
    const int c = threadIdx.x & 3;
    const int tiles = (s.T + kRowsPerBlock - 1) / kRowsPerBlock;
    const int bhk = blockIdx.x / tiles;               // b * Hkv + hk
    const int j = (blockIdx.x % tiles) * kRowsPerBlock + (threadIdx.x >> 2);
    const int b = bhk / s.Hkv, hk = bhk % s.Hkv;
    const bool kvalid = j < s.T;
    const int jj = kvalid ? j : s.T - 1;

    float2 dk2[8], dv2[8], x[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) { dk2[e] = make_float2(0.f, 0.f); dv2[e] = make_float2(0.f, 0.f); }

    for (int g = 0; g < s.G; ++g) {
        const int bh = b * s.H + hk * s.G + g;
        using R = typename RotOf<T>::type;
        const R* Qt = reinterpret_cast<const R*>(a.qt) + ((size_t)bh * s.T) * kHeadDim;
        const T* dO = reinterpret_cast<const T*>(a.dout) + ((size_t)bh * s.T) * kHeadDim;
        const float* P = a.P + (size_t)bh * s.T * a.S;
        const float* DP = a.DP + (size_t)bh * s.T * a.S;
        const float* Dl = a.Delta + (size_t)bh * s.T;
        for (int t = 0; t <= s.W; ++t) {
            const int i = jj + t;
            const bool ok = i < s.T;
            const int ic = ok ? i : jj;
            const float p = ok ? P[(size_t)ic * a.S + t] : 0.f;
            const float ds = ok ? p * (DP[(size_t)ic * a.S + t] - Dl[ic]) * s.scale : 0.f;
            load_chunk2(Qt + (size_t)ic * kHeadDim, c, x);
            axpy16x2(ds, x, dk2);
            load_chunk2(dO + (size_t)ic * kHeadDim, c, x);
            axpy16x2(p, x, dv2);
            if (__all_sync(0xffffffffu, !ok)) break;
        }
        for (int k = 0; k < a.r.K; ++k) {
            if (!((a.r.active >> k) & 1u)) continue;
            const int slot = s.W + 1 + k;
            const float w = a.r.w[k];
#pragma unroll
            for (int side = 0; side < 2; ++side) {
                const float cw = side == 0 ? 1.f - w : w;
                if (side == 1 && w == 0.f) break;       // warp-uniform
                const long long il = (long long)jj + a.r.s0[k] + side;
                const bool ok = il < s.T;
                const int ic = ok ? (int)il : jj;
                const float pr = ok ? P[(size_t)ic * a.S + slot] : 0.f;
                const float ds = ok ? pr * (DP[(size_t)ic * a.S + slot] - Dl[ic]) * s.scale * cw : 0.f;
                const float p = pr * cw;
                if (__all_sync(0xffffffffu, !ok)) continue;
                load_chunk2(Qt + (size_t)ic * kHeadDim, c, x);
                axpy16x2(ds, x, dk2);
                load_chunk2(dO + (size_t)ic * kHeadDim, c, x);
                axpy16x2(p, x, dv2);
            }
        }
    }
    float dk[16], dv[16];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        dk[2 * e] = dk2[e].x; dk[2 * e + 1] = dk2[e].y;
        dv[2 * e] = dv2[e].x; dv[2 * e + 1] = dv2[e].y;
    }
    if (kvalid) {
        rope_chunk(a.rope, jj, c, dk, true);
        const size_t off = ((size_t)bhk * s.T + j) * kHeadDim;
        store_chunk(reinterpret_cast<T*>(a.dk) + off, c, dk);
        store_chunk(reinterpret_cast<T*>(a.dv) + off, c, dv);
    }
}

}  // namespace

cudaError_t launch_rope_rows(const void* src, void* dst, long long rows, int T, const RopeParams& rp,
                             bool bf16, cudaStream_t st, unsigned* status) {
    if (rows <= 0) return cudaSuccess;
    const long long items = rows * 4;
    long long grid = (items + 255) / 256;
    if (grid > 152 * 16) grid = 152 * 16;       // 16 resident 256-thread blocks on each of 152 SMs
    if (bf16) {
        const int heads = (int)(rows / T);
        // one tile per block (the hardware hands the blocks to the SMs as
        // they free up, which balances the load better than a grid-stride
        // loop); tiles of 32 heads while they still give two blocks per SM,
        // else of 16 (B16 H8 T1024: 2.296 -> 2.281 ms per 16-layer step;
        // with two kv heads, 512 tiles of 16 heads beat 128 of 32)
        static int sms = 0;
        if (sms == 0) {
            int dev = 0;
            if (cudaGetDevice(&dev) != cudaSuccess ||
                cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
                sms = 152;
        }
        const long long tp = (T + kRopePos - 1) / kRopePos;
        const long long t32 = tp * ((heads + 31) / 32), t16 = tp * ((heads + 15) / 16);
        const __nv_bfloat16* s16 = reinterpret_cast<const __nv_bfloat16*>(src);
        __half* d16 = reinterpret_cast<__half*>(dst);
        if (t32 >= 2LL * sms)
            return launch_kernel(rope_rows_bf16_kernel<32>, dim3((unsigned)std::min(t32, 0x7fffffffLL)), dim3(256),
                                 0, st, s16, d16, heads, T, rp, status);
        return launch_kernel(rope_rows_bf16_kernel<16>, dim3((unsigned)std::min(t16, 0x7fffffffLL)), dim3(256), 0,
                             st, s16, d16, heads, T, rp, status);
    }
    return launch_kernel(rope_rows_kernel<float, float>, dim3((unsigned)grid), dim3(256), 0, st,
                         reinterpret_cast<const float*>(src), reinterpret_cast<float*>(dst), rows, T, rp);
}

cudaError_t launch_fwd_simple(const FwdArgs& a, bool bf16, cudaStream_t st) {
    const long long tiles = (a.s.T + kRowsPerBlock - 1) / kRowsPerBlock;
    const long long grid = tiles * a.s.B * a.s.H;
    if (grid <= 0) return cudaSuccess;
    if (bf16) return launch_kernel(fwd_simple_kernel<__nv_bfloat16>, dim3((unsigned)grid), dim3(kThreads), 0, st, a);
    return launch_kernel(fwd_simple_kernel<float>, dim3((unsigned)grid), dim3(kThreads), 0, st, a);
}

int bwd_simple_blocks(const Shape& s) {
    const long long tiles = (s.T + kRowsPerBlock - 1) / kRowsPerBlock;
    return (int)(tiles * s.B * s.H);
}

cudaError_t launch_bwd_query(const BwdArgs& a, bool bf16, cudaStream_t st) {
    const long long tiles = (a.s.T + kRowsPerBlock - 1) / kRowsPerBlock;
    const long long gq = tiles * a.s.B * a.s.H;
    if (gq <= 0) return cudaSuccess;
    if (bf16) return launch_kernel(bwd_query_kernel<__nv_bfloat16>, dim3((unsigned)gq), dim3(kThreads), 0, st, a);
    return launch_kernel(bwd_query_kernel<float>, dim3((unsigned)gq), dim3(kThreads), 0, st, a);
}

cudaError_t launch_bwd_key(const BwdArgs& a, bool bf16, cudaStream_t st) {
    const long long tiles = (a.s.T + kRowsPerBlock - 1) / kRowsPerBlock;
    const long long gk = tiles * a.s.B * a.s.Hkv;
    if (gk <= 0) return cudaSuccess;
    if (bf16) return launch_kernel(bwd_key_kernel<__nv_bfloat16>, dim3((unsigned)gk), dim3(kThreads), 0, st, a);
    return launch_kernel(bwd_key_kernel<float>, dim3((unsigned)gk), dim3(kThreads), 0, st, a);
}

}  // namespace fibattn
