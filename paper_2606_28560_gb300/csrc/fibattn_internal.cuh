// fibattn_internal.cuh -- shared definitions of the CUDA library (not part of
// the C ABI).  Depth-staggered scaled-Fibonacci sparse attention,
// arXiv 2606.28560, Section 2.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

namespace fibattn {

constexpr int kHeadDim = 64;      // D; every kernel is specialised for it
constexpr int kHalf = kHeadDim / 2;
constexpr int kMaxRungs = 32;     // K limit of the ABI
constexpr int kMaxWindow = 1024;  // W limit of the ABI

// Per-rung data prepared on the host (Section 2: d_k = alpha * f_k, read by
// linear interpolation between the floor and floor-plus-one rows).
struct RungParams {
    int K;                    // number of rungs passed by the caller
    unsigned active;          // bit k: rung k can ever be attended (dedup, reach)
    int s0[kMaxRungs];        // floor(d_k)
    float w[kMaxRungs];       // d_k - floor(d_k): weight of the far row i-s0-1
    float d[kMaxRungs];       // d_k in fp32; the rung is masked for queries i < d_k
    float f[kMaxRungs];       // base value f_k (for dL/dalpha = sum_k f_k dL/dd_k)
};

// RoPE phase increments: the rotation angle of pair m at position p is
// 2*pi * frac(p * F[m] / 2^64), F[m] = round(2^64 * theta_m / (2*pi)),
// theta_m = base^(-2m/D).  The integer product wraps modulo one turn exactly,
// so the angle is reduced without any floating-point range reduction.
struct RopeParams {
    unsigned long long F[kHalf];
};

// Division by a divisor fixed at launch, for numerators below 2^31: the
// quotient is (umulhi(n, mul) + n) >> shift with shift = ceil(log2 d) and
// mul = floor(2^32 (2^shift - d) / d) + 1 (the round-up multiplier method).
struct FastDiv {
    unsigned d, mul, shift;
#ifdef __CUDACC__
    __host__ __device__
#endif
    static FastDiv make(unsigned d) {
        FastDiv f;
        f.d = d;
        f.shift = 0;
        while ((1ull << f.shift) < d) ++f.shift;
        f.mul = (unsigned)(((1ull << 32) * ((1ull << f.shift) - d)) / d + 1);
        return f;
    }
};
#ifdef __CUDACC__
__device__ __forceinline__ unsigned fdiv(unsigned n, const FastDiv& f) {
    return (__umulhi(n, f.mul) + n) >> f.shift;
}
#endif

struct Shape {
    int B, H, Hkv, T, W, G;   // G = H / Hkv
    float scale;              // score scale (1/sqrt(D) by default)
    FastDiv dH, dHkv, dG, dTiles;   // by H, Hkv, G and the tensor-core tiles per head
};

// Device status word (one per device, read and cleared by
// fibattn_check_status): kernels OR these bits into it.
constexpr unsigned kStatusWaitTimeout = 1u;   // a bounded wait on a staging copy ran out
constexpr unsigned kStatusRange = 2u;         // a rotated row overflowed its fp16 storage
__device__ __forceinline__ void raise_status(unsigned* st, unsigned bits) {
    if (st) atomicOr(st, bits);
}

struct FwdArgs {
    const void* q;            // [B,H,T,D]
    const void* kt;           // rotated keys [B,Hkv,T,D] (workspace)
    const void* k;            // raw keys (prologue input)
    const void* v;            // [B,Hkv,T,D]
    void* out;                // [B,H,T,D]
    float* lse;               // [B,H,T]
    // Optional residuals for the backward (tensor-core forward only; all
    // nullptr when not asked for): the rotated queries, the unnormalised
    // probability exp(s - max) of every slot (0 where not attended), the
    // far-minus-floor raw score of every rung row and 1 / (row sum) per query.
    void* res_qt;             // bf16 [B,H,T,D]
    float* res_P;             // slot-major [B,H,S,T], S = W + 1 + K
    float* res_sd;            // rung-major [B,H,K,T]
    float* res_il;            // [B,H,T]
    unsigned* status;         // device status word
    int S;
    Shape s;
    RungParams r;
    RopeParams rope;
};

struct BwdArgs {
    const void* q;            // [B,H,T,D]
    const void* k;            // [B,Hkv,T,D]
    const void* v;
    const float* lse;         // [B,H,T]
    const void* dout;         // [B,H,T,D]
    const void* out;          // forward output [B,H,T,D] or nullptr
    void* dq;                 // [B,H,T,D]
    void* dk;                 // [B,Hkv,T,D]
    void* dv;
    float* dtheta;            // device scalar or nullptr
    int want_dd;              // compute dL/dd_k (dtheta or dd requested)
    float* dd;                // device [K] or nullptr
    // workspace views
    void* qt;                 // rotated q [B,H,T,D] (bf16 from the tensor-core query pass, fp16 from the prologue)
    void* kt;                 // rotated k [B,Hkv,T,D]
    float* P;                 // softmax probabilities [B,H,T,S]
    float* DP;                // dL/dp = dO . val per slot [B,H,T,S]
    float* Delta;             // sum_slots p dL/dp per query [B,H,T]
    float* Ps;                // tensor-core path, slot-major [B,H,S,T]: p      (P region)
    float* DSs;               //                                      dS = p (dp - Delta)  (DP region)
    long long* rpart;         // per query-pass block dL/dd_k partials, 2^-32 fixed point [kMaxRungs][nblk_q]
    const float* res_il;      // forward residual 1 / (row sum) [B,H,T] (p = Ps[slot] * res_il)
    const float* res_sd;      // forward residual far-minus-floor rung scores [B,H,K,T], or nullptr;
                              // when the forward residuals are used, Ps and qt point into them
    int saved;                // tensor-core passes read p (Ps, unnormalised), sd and q~ (qt) from the forward residuals
    unsigned* status;         // device status word
    int nblk_q;               // query-pass blocks
    int S;                    // slots per query = W + 1 + K
    float alpha;
    Shape s;
    RungParams r;
    RopeParams rope;
};

// ---------------------------------------------------------------- RoPE ----

// cos/sin of the angle of pair m at position pos (see RopeParams).
__device__ __forceinline__ void rope_cs(const RopeParams& rp, int m, int pos, float& c, float& s) {
    unsigned long long ph = (unsigned long long)(unsigned)pos * rp.F[m];
    int hi = (int)(unsigned)(ph >> 32);              // signed turn fraction in [-1/2, 1/2)
    float ang = (float)hi * 1.4629180792671596e-09f; // 2*pi / 2^32
    __sincosf(ang, &s, &c);
}

// ------------------------------------------------------------- element IO --

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T> struct Vec8;   // 8 consecutive elements

template <> struct Vec8<float> {
    static __device__ __forceinline__ void load(const float* p, float* x) {
        float4 a = *reinterpret_cast<const float4*>(p);
        float4 b = *reinterpret_cast<const float4*>(p + 4);
        x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w; x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
    }
    static __device__ __forceinline__ void store(float* p, const float* x) {
        *reinterpret_cast<float4*>(p) = make_float4(x[0], x[1], x[2], x[3]);
        *reinterpret_cast<float4*>(p + 4) = make_float4(x[4], x[5], x[6], x[7]);
    }
};

template <> struct Vec8<__nv_bfloat16> {
    static __device__ __forceinline__ void load(const __nv_bfloat16* p, float* x) {
        uint4 u = *reinterpret_cast<const uint4*>(p);
        unsigned w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            x[2 * i] = __uint_as_float(w[i] << 16);
            x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
        }
    }
    static __device__ __forceinline__ void store(__nv_bfloat16* p, const float* x) {
        uint4 u;
        unsigned w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            __nv_bfloat162 h = __floats2bfloat162_rn(x[2 * i], x[2 * i + 1]);
            w[i] = *reinterpret_cast<unsigned*>(&h);
        }
        u.x = w[0]; u.y = w[1]; u.z = w[2]; u.w = w[3];
        *reinterpret_cast<uint4*>(p) = u;
    }
};

// fp16 holds the RoPE-rotated q/k rows of the bf16 path: 10 mantissa bits
// against bf16's 7 keep the score error well inside the bf16 tolerance.
template <> struct Vec8<__half> {
    static __device__ __forceinline__ void load(const __half* p, float* x) {
        uint4 u = *reinterpret_cast<const uint4*>(p);
        unsigned w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float2 f = __half22float2(*reinterpret_cast<__half2*>(&w[i]));
            x[2 * i] = f.x;
            x[2 * i + 1] = f.y;
        }
    }
    static __device__ __forceinline__ void store(__half* p, const float* x) {
        uint4 u;
        unsigned w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            __half2 h = __floats2half2_rn(x[2 * i], x[2 * i + 1]);
            w[i] = *reinterpret_cast<unsigned*>(&h);
        }
        u.x = w[0]; u.y = w[1]; u.z = w[2]; u.w = w[3];
        *reinterpret_cast<uint4*>(p) = u;
    }
};

// Storage type of rotated rows: fp32 for fp32 I/O, fp16 for bf16 I/O.
template <typename T> struct RotOf { using type = float; };
template <> struct RotOf<__nv_bfloat16> { using type = __half; };

// A lane of a 4-lane group owns RoPE pairs [8c, 8c+8): head dims 8c..8c+7
// (x[0..7]) and 32+8c..32+8c+7 (x[8..15]), so a rotation stays in the lane.
template <typename T>
__device__ __forceinline__ void load_chunk(const T* row, int c, float* x) {
    Vec8<T>::load(row + 8 * c, x);
    Vec8<T>::load(row + kHalf + 8 * c, x + 8);
}
template <typename T>
__device__ __forceinline__ void store_chunk(T* row, int c, const float* x) {
    Vec8<T>::store(row + 8 * c, x);
    Vec8<T>::store(row + kHalf + 8 * c, x + 8);
}

// x <- R(pos) x (inverse = false) or R(pos)^T x (inverse = true) for the 8
// pairs owned by lane c.
__device__ __forceinline__ void rope_chunk(const RopeParams& rp, int pos, int c, float* x, bool inverse) {
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        float cs, sn;
        rope_cs(rp, 8 * c + u, pos, cs, sn);
        if (inverse) sn = -sn;
        float a = x[u], b = x[8 + u];
        x[u] = a * cs - b * sn;
        x[8 + u] = b * cs + a * sn;
    }
}

// ------------------------------------------------- rung-gradient reduction --

// dL/dd_k is the sum of the query blocks' partials.  Each block writes its
// partials as 64-bit fixed point (2^-32 units; threads k < K hold rung k's);
// block 0 of the key pass, which starts after the query pass has completed,
// adds them up -- integer addition is exact and order-free, so the result
// does not depend on scheduling -- and applies the chain rule
// dL/dalpha = sum_k f_k dL/dd_k, dL/dtheta = dL/dalpha (alpha - 0.5)(1.5 - alpha),
// alpha = 0.5 + sigmoid(theta).
__device__ __forceinline__ void write_rung_partials(const BwdArgs& a, float partial) {
    if ((int)threadIdx.x < a.r.K)
        a.rpart[(size_t)threadIdx.x * a.nblk_q + blockIdx.x] = __float2ll_rn(partial * 4294967296.0f);
}

// Called by every thread of block 0 of the key pass (blockDim a multiple of
// 32, at most 32 warps).  red: shared scratch of at least K floats; red64:
// shared scratch of at least (blockDim / 32) * K 64-bit words.
__device__ __forceinline__ void convert_rung_sums(const BwdArgs& a, float* red, long long* red64) {
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5, nw = blockDim.x >> 5;
    for (int k = 0; k < a.r.K; ++k) {
        const long long* col = a.rpart + (size_t)k * a.nblk_q;
        long long v = 0;
        for (int blk = t; blk < a.nblk_q; blk += blockDim.x) v += __ldcg(col + blk);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) red64[warp * a.r.K + k] = v;
    }
    __syncthreads();
    if (t < a.r.K) {
        long long tot = 0;
        for (int w = 0; w < nw; ++w) tot += red64[w * a.r.K + t];
        const float v = (float)((double)tot * 2.3283064365386962890625e-10);
        red[t] = v;
        if (a.dd) a.dd[t] = v;
    }
    __syncthreads();
    if (t == 0 && a.dtheta) {
        float da = 0.f;
        for (int k = 0; k < a.r.K; ++k) da += a.r.f[k] * red[k];
        *a.dtheta = da * (a.alpha - 0.5f) * (1.5f - a.alpha);
    }
}

// ------------------------------------------- programmatic dependent launch --

// Every kernel starts with this, before its first global-memory access: it
// waits until the previous kernel in the stream has completed and its writes
// are visible (a no-op when the launch carries no programmatic dependency),
// then lets the next kernel be scheduled, so that its blocks can become
// resident and run up to their own wait while this grid's last blocks run.
__device__ __forceinline__ void grid_dependency_sync() {
    asm volatile("griddepcontrol.wait;\n" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}
// The two halves, for a kernel that knows which of its inputs the kernel
// before it (launched by the same library call) does not write: it lets the
// next launch be scheduled at once, reads those inputs, and waits only before
// touching anything the previous kernel may produce.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }

// Host: whether launches carry the programmatic-serialisation attribute
// (environment FIBATTN_PDL=0 turns it off).
bool pdl_enabled();

template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                          Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 1 : 0;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, args...);
    return e != cudaSuccess ? e : cudaGetLastError();
}

// ----------------------------------------------------------- launchers ----

cudaError_t launch_rope_rows(const void* src, void* dst, long long rows, int T, const RopeParams& rp,
                             bool bf16, cudaStream_t st, unsigned* status);
cudaError_t launch_fwd_simple(const FwdArgs& a, bool bf16, cudaStream_t st);
cudaError_t launch_bwd_query(const BwdArgs& a, bool bf16, cudaStream_t st);
cudaError_t launch_bwd_key(const BwdArgs& a, bool bf16, cudaStream_t st);
int bwd_simple_blocks(const Shape& s);

// Records a message for fibattn_last_error() and returns `code`.
int set_error(int code, const char* msg);

// Opt-in per-kernel timing: when enabled, each launch is bracketed by CUDA
// events recorded on the caller's stream (see fibattn_profile_* in the ABI).
struct ProfScope {
    ProfScope(const char* name, cudaStream_t st);
    ~ProfScope();
    const char* name_;
    cudaStream_t st_;
    cudaEvent_t start_;
    bool on_;
};

}  // namespace fibattn
