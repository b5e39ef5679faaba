// fibattn_api.cu -- the C ABI declared in include/fibattn.h: argument checks,
// host-side parameter prep (rung distances, RoPE phase increments),
// workspace layout, and the launches.  arXiv 2606.28560, Section 2.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <cstdint>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/fibattn.h"
#include "fibattn_internal.cuh"
#include "fwd_mma.cuh"
#include "mma_common.cuh"

using namespace fibattn;

namespace {
// The device status word that kernels OR kStatus* bits into (one per device:
// every device that loads the library holds its own copy).  Host code looks
// up its device address once per device, with that device current.
__device__ unsigned g_status_word;
}  // namespace

namespace fibattn {
bool pdl_enabled() {
    static const bool on = [] {
        const char* v = std::getenv("FIBATTN_PDL");
        return !(v && v[0] == '0');
    }();
    return on;
}
}  // namespace fibattn

namespace {

thread_local std::string g_err;

int fail(int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_err = buf;
    return code;
}

size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// rotated q/k rows in the workspace: fp32 (fp32 I/O) or fp16 (bf16 I/O)
size_t rot_size(int dtype) { return dtype == FIBATTN_BF16 ? 2 : 4; }

struct Resolved {
    float rope_base, scale;
    int Hkv, dedup, round_offsets, fwd_kernel, bwd_kernel;
    void* rotated_k;
    void* residuals;
};

int resolve_opts(const fibattn_opts* o, int H, int D, Resolved* r) {
    r->rope_base = (o && o->rope_base != 0.f) ? o->rope_base : 1e4f;
    r->scale = (o && o->scale > 0.f) ? o->scale : (float)(1.0 / std::sqrt((double)D));
    r->Hkv = (o && o->Hkv > 0) ? o->Hkv : H;
    r->dedup = (o && o->no_dedup) ? 0 : 1;
    r->round_offsets = (o && o->round_offsets) ? 1 : 0;
    r->fwd_kernel = o ? o->fwd_kernel : 0;
    if (r->fwd_kernel < 0 || r->fwd_kernel > 3) return fail(FIBATTN_ERR_INVALID_ARG, "fwd_kernel must be 0, 1, 2 or 3");
    r->bwd_kernel = o ? o->bwd_kernel : 0;
    r->rotated_k = o ? o->rotated_k : nullptr;
    if ((uintptr_t)r->rotated_k & 15u) return fail(FIBATTN_ERR_INVALID_ARG, "rotated_k must be 16-byte aligned");
    r->residuals = o ? o->residuals : nullptr;
    if ((uintptr_t)r->residuals & 15u) return fail(FIBATTN_ERR_INVALID_ARG, "residuals must be 16-byte aligned");
    if (r->bwd_kernel < 0 || r->bwd_kernel > 2) return fail(FIBATTN_ERR_INVALID_ARG, "bwd_kernel must be 0, 1 or 2");
    if (!(r->rope_base > 1.f) || !std::isfinite(r->rope_base))
        return fail(FIBATTN_ERR_INVALID_ARG, "rope_base must be finite and > 1 (got %g)", (double)r->rope_base);
    if (!std::isfinite(r->scale)) return fail(FIBATTN_ERR_INVALID_ARG, "scale must be finite");
    if (r->Hkv <= 0 || H % r->Hkv) return fail(FIBATTN_ERR_INVALID_ARG, "H (%d) must be a multiple of Hkv (%d)", H, r->Hkv);
    return FIBATTN_OK;
}

int check_shape(int B, int H, int T, int D, int W, int K, int dtype) {
    if (dtype != FIBATTN_F32 && dtype != FIBATTN_BF16) return fail(FIBATTN_ERR_INVALID_ARG, "unknown dtype %d", dtype);
    if (B < 0 || H <= 0 || T < 1 || T > (1 << 20)) return fail(FIBATTN_ERR_INVALID_ARG, "bad shape B=%d H=%d T=%d", B, H, T);
    if (D != kHeadDim) return fail(FIBATTN_ERR_UNSUPPORTED, "only D == %d is built (got %d)", kHeadDim, D);
    if (W < 0 || W > kMaxWindow) return fail(FIBATTN_ERR_INVALID_ARG, "W must be in [0, %d] (got %d)", kMaxWindow, W);
    if (K < 0 || K > kMaxRungs) return fail(FIBATTN_ERR_INVALID_ARG, "K must be in [0, %d] (got %d)", kMaxRungs, K);
    if ((long long)B * H * T > (1LL << 31) / 64) return fail(FIBATTN_ERR_INVALID_ARG, "B*H*T too large");
    return FIBATTN_OK;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// Section 2: d_k = alpha f_k, rounded once to fp32; s0 = floor(d_k), w = d_k - s0.
// round_offsets: the integer-offset variants of the paper's boolean-mask path
// (Section 2, "Implementation note"): d_k is then rounded half to even to an
// integer after the fp32 product, so every rung reads one row (w = 0).
int prep_rungs(float alpha, const float* f, int K, int W, int dedup, int T, RungParams* r, int round_offsets = 0) {
    if (!(alpha >= 0.5f && alpha <= 1.5f)) return fail(FIBATTN_ERR_INVALID_ARG, "alpha must be in [0.5, 1.5] (got %g)", (double)alpha);
    if (K > 0 && !f) return fail(FIBATTN_ERR_INVALID_ARG, "offsets is NULL");
    std::memset(r, 0, sizeof(*r));
    r->K = K;
    for (int k = 0; k < K; ++k) {
        if (!std::isfinite(f[k]) || f[k] < 0.f) return fail(FIBATTN_ERR_INVALID_ARG, "offsets[%d] must be finite and >= 0", k);
        volatile float d = alpha * f[k];        // one fp32 rounding
        if (!std::isfinite(d)) return fail(FIBATTN_ERR_INVALID_ARG, "alpha*offsets[%d] overflows", k);
        if (round_offsets) d = std::nearbyint((float)d);   // to nearest, ties to even (default mode)
        r->f[k] = f[k];
        r->d[k] = d;
        bool reach = d <= (float)(T - 1);       // otherwise masked for every query
        bool keep = dedup ? (d > (float)W) : true;
        if (reach && keep) {
            float fl = std::floor(d);
            r->s0[k] = (int)fl;
            r->w[k] = d - fl;                   // exact in fp32
            r->active |= 1u << k;
        } else {
            r->s0[k] = 0;
            r->w[k] = 0.f;
        }
    }
    return FIBATTN_OK;
}

// F[m] = round(2^64 * theta_m / (2 pi)), theta_m = base^(-2m/D)  (fp64 on the host)
void prep_rope(float base, RopeParams* rp) {
    const double two_pi = 6.283185307179586476925286766559;
    for (int m = 0; m < kHalf; ++m) {
        double theta = std::pow((double)base, -2.0 * m / (double)kHeadDim);
        double frac = theta / two_pi;           // in (0, 1)
        long double scaled = std::ldexp((long double)frac, 64);
        rp->F[m] = (unsigned long long)(scaled + 0.5L);
    }
}

Shape make_shape(int B, int H, int T, int W, const Resolved& o) {
    Shape s;
    s.B = B; s.H = H; s.Hkv = o.Hkv; s.T = T; s.W = W; s.G = H / o.Hkv; s.scale = o.scale;
    s.dH = FastDiv::make((unsigned)H);
    s.dHkv = FastDiv::make((unsigned)o.Hkv);
    s.dG = FastDiv::make((unsigned)s.G);
    s.dTiles = FastDiv::make((unsigned)((T + kMmaTile - 1) / kMmaTile));
    return s;
}

// Forward residuals (fibattn_opts.residuals): rotated q (bf16), unnormalised
// p per slot (slot-major), far-minus-floor rung scores (rung-major), 1 / (row
// sum) per query.
struct ResLayout {
    size_t qt, P, sd, il, total;
};

ResLayout res_layout(int B, int H, int T, int W, int K) {
    ResLayout L;
    const size_t n = (size_t)B * H * T;
    L.qt = 0;
    L.P = align256(n * kHeadDim * 2);
    L.sd = L.P + align256(n * ((size_t)W + 1 + K) * 4);
    L.il = L.sd + align256(n * (size_t)K * 4);
    L.total = L.il + align256(n * 4);
    return L;
}

struct BwdLayout {
    size_t qt, kt, P, DP, Delta, rpart, total;
};

BwdLayout bwd_layout(int B, int H, int Hkv, int T, int W, int K, int dtype, bool own_kt) {
    BwdLayout L;
    size_t es = rot_size(dtype);
    size_t S = (size_t)W + 1 + K;
    size_t off = 0;
    L.qt = off; off += align256((size_t)B * H * T * kHeadDim * es);
    L.kt = off;
    if (own_kt) off += align256((size_t)B * Hkv * T * kHeadDim * es);   // else the caller's rotated_k
    L.P = off; off += align256((size_t)B * H * T * S * 4);
    L.DP = off; off += align256((size_t)B * H * T * S * 4);
    L.Delta = off; off += align256((size_t)B * H * T * 4);
    L.rpart = off;                                  // fixed-point rung partials, one per query block
    Shape s;
    std::memset(&s, 0, sizeof(s));
    s.B = B; s.H = H; s.Hkv = Hkv; s.T = T; s.W = W; s.G = H / Hkv;
    off += align256((size_t)kMaxRungs * 8 * std::max(bwd_simple_blocks(s), bwd_mma_blocks(s)));
    L.total = off;
    return L;
}

int cuda_fail(cudaError_t e, const char* what) {
    return fail(FIBATTN_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Device address of the current device's status word (looked up once per
// device; no allocation).
constexpr int kMaxDevices = 256;
std::mutex g_status_mu;
unsigned* g_status_addr[kMaxDevices];

int status_word(unsigned** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(FIBATTN_ERR_CUDA, "device ordinal %d out of range", dev);
    std::lock_guard<std::mutex> g(g_status_mu);
    if (!g_status_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_status_word);
        if (e != cudaSuccess || !p) return cuda_fail(e, "cudaGetSymbolAddress of the status word");
        g_status_addr[dev] = static_cast<unsigned*>(p);
    }
    *out = g_status_addr[dev];
    return FIBATTN_OK;
}

// Test hook: one warp arms an mbarrier for 128 bytes that no copy will
// deliver and waits on it with the library's bounded wait, so the wait runs
// out after limit_ns and raises kStatusWaitTimeout (nothing is ever written
// into the barrier's transaction count, so nothing is left in flight).
__global__ void wait_timeout_probe_kernel(unsigned* status, unsigned long long limit_ns) {
    __shared__ unsigned long long bar;
    if (threadIdx.x == 0) {
        mma::mbar_init(&bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    }
    __syncwarp();
    if (threadIdx.x == 0) mma::mbar_expect_tx(&bar, 128u);
    __syncwarp();
    const bool ok = mma::mbar_wait(&bar, 0, limit_ns);
    if (!ok && threadIdx.x == 0) raise_status(status, kStatusWaitTimeout);
}

// Tensor maps are encoded through the driver, which needs a current context,
// and a host thread that has made no runtime call yet (e.g. a framework's
// backward worker) has none: make the primary context of the thread's current
// device current before the first encode or launch.
int bind_context() {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaSetDevice(dev);
    return e == cudaSuccess ? FIBATTN_OK : cuda_fail(e, "binding the current device's context");
}

// ---------------------------------------------------------------- profiler --

struct ProfRecord { std::string name; cudaEvent_t a, b; };
std::mutex g_prof_mu;
bool g_prof_on = false;
std::vector<ProfRecord> g_prof_recs;
std::vector<cudaEvent_t> g_prof_pool;

cudaEvent_t prof_event() {
    cudaEvent_t e = nullptr;
    if (!g_prof_pool.empty()) { e = g_prof_pool.back(); g_prof_pool.pop_back(); return e; }
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

}  // namespace

namespace fibattn {
int set_error(int code, const char* msg) { return fail(code, "%s", msg); }

// During stream capture the records become external event nodes of the
// graph, so every replay of the graph re-times the kernel.
static cudaError_t prof_record(cudaEvent_t e, cudaStream_t st) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive)
        return cudaEventRecordWithFlags(e, st, cudaEventRecordExternal);
    return cudaEventRecord(e, st);
}

ProfScope::ProfScope(const char* name, cudaStream_t st) : name_(name), st_(st), start_(nullptr), on_(false) {
    std::lock_guard<std::mutex> g(g_prof_mu);
    if (!g_prof_on) return;
    start_ = prof_event();
    if (start_ && prof_record(start_, st_) == cudaSuccess) on_ = true;
}
ProfScope::~ProfScope() {
    if (!on_) return;
    std::lock_guard<std::mutex> g(g_prof_mu);
    cudaEvent_t b = prof_event();
    if (b && prof_record(b, st_) == cudaSuccess) g_prof_recs.push_back({name_, start_, b});
}
}  // namespace fibattn

extern "C" {

int fibattn_profile_enable(int on) {
    std::lock_guard<std::mutex> g(g_prof_mu);
    g_prof_on = on != 0;
    for (auto& r : g_prof_recs) { g_prof_pool.push_back(r.a); g_prof_pool.push_back(r.b); }
    g_prof_recs.clear();
    // create the events up front so that recording during a timed region
    // costs no event creation on the host
    const size_t kPool = 1 << 14;
    while (g_prof_on && g_prof_pool.size() < kPool) {
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) break;
        g_prof_pool.push_back(e);
    }
    g_prof_recs.reserve(kPool / 2);
    return FIBATTN_OK;
}

int fibattn_profile_summary(int index, char* name, int name_len, double* total_ms, int* launches) {
    std::lock_guard<std::mutex> g(g_prof_mu);
    std::vector<std::string> names;
    for (auto& r : g_prof_recs) {
        bool seen = false;
        for (auto& n : names) seen = seen || n == r.name;
        if (!seen) names.push_back(r.name);
    }
    if (index < 0) return (int)names.size();
    if (index >= (int)names.size()) return fail(FIBATTN_ERR_INVALID_ARG, "profile index out of range");
    double tot = 0.0;
    int cnt = 0;
    for (auto& r : g_prof_recs) {
        if (r.name != names[index]) continue;
        cudaError_t e = cudaEventSynchronize(r.b);
        if (e != cudaSuccess) return cuda_fail(e, "profile event sync");
        float ms = 0.f;
        e = cudaEventElapsedTime(&ms, r.a, r.b);
        if (e != cudaSuccess) return cuda_fail(e, "profile elapsed time");
        tot += ms;
        ++cnt;
    }
    if (name && name_len > 0) { std::strncpy(name, names[index].c_str(), name_len - 1); name[name_len - 1] = 0; }
    if (total_ms) *total_ms = tot;
    if (launches) *launches = cnt;
    return FIBATTN_OK;
}

const char* fibattn_last_error(void) { return g_err.c_str(); }

size_t fibattn_residual_bytes(int B, int H, int T, int D, int W, int K, int dtype) {
    if (check_shape(B, H, T, D, W, K, dtype) || dtype != FIBATTN_BF16) return 0;
    return res_layout(B, H, T, W, K).total;
}

int fibattn_rung_params(float alpha, const float* offsets, int K, int W, int no_dedup, int round_offsets,
                        float* d, int* s0, float* w, int* active) {
    if (K < 0 || K > kMaxRungs) return fail(FIBATTN_ERR_INVALID_ARG, "K must be in [0, %d]", kMaxRungs);
    if (W < 0) return fail(FIBATTN_ERR_INVALID_ARG, "W must be >= 0");
    RungParams r;
    int rc = prep_rungs(alpha, offsets, K, W, no_dedup ? 0 : 1, 1 << 30, &r, round_offsets);
    if (rc) return rc;
    for (int k = 0; k < K; ++k) {
        if (d) d[k] = r.d[k];
        float fl = std::floor(r.d[k]);
        if (s0) s0[k] = (int)fl;
        if (w) w[k] = r.d[k] - fl;
        if (active) active[k] = (r.active >> k) & 1u;
    }
    return FIBATTN_OK;
}

int fibattn_base(int kind, int K, float* f) {
    if (!f || K < 0 || K > 64) return fail(FIBATTN_ERR_INVALID_ARG, "bad arguments to fibattn_base");
    if (kind == 0) {                            // Fibonacci 1, 2, 3, 5, ...
        double a = 1, b = 2;
        for (int k = 0; k < K; ++k) { f[k] = (float)a; double n = a + b; a = b; b = n; }
    } else if (kind == 1) {                     // powers of two
        for (int k = 0; k < K; ++k) f[k] = std::ldexp(1.f, k);
    } else {
        return fail(FIBATTN_ERR_INVALID_ARG, "unknown base kind %d", kind);
    }
    return FIBATTN_OK;
}

int fibattn_alpha_schedule(int kind, int L, const float* theta, int stride, float* alpha) {
    if (!alpha || L < 1) return fail(FIBATTN_ERR_INVALID_ARG, "bad arguments to fibattn_alpha_schedule");
    for (int l = 0; l < L; ++l) {
        switch (kind) {
        case 0: alpha[l] = 1.f; break;
        case 1:
            if (!theta) return fail(FIBATTN_ERR_INVALID_ARG, "learned schedule needs theta");
            alpha[l] = (float)(0.5 + 1.0 / (1.0 + std::exp(-(double)theta[l])));
            break;
        case 2: alpha[l] = L > 1 ? (float)(0.5 + (double)l / (L - 1)) : 1.f; break;
        case 3: {
            int a = stride, b = L;              // gcd(stride, L) must be 1
            while (b) { int t = a % b; a = b; b = t; }
            if (stride <= 0 || a != 1) return fail(FIBATTN_ERR_INVALID_ARG, "stride %d not coprime to L=%d", stride, L);
            int idx = (int)(((long long)stride * l) % L);
            alpha[l] = L > 1 ? (float)(0.5 + (double)idx / (L - 1)) : 1.f;
            break;
        }
        default: return fail(FIBATTN_ERR_INVALID_ARG, "unknown schedule kind %d", kind);
        }
    }
    return FIBATTN_OK;
}

int fibattn_theta_of_alpha(int L, const float* alpha, float* theta) {
    if (!alpha || !theta || L < 1) return fail(FIBATTN_ERR_INVALID_ARG, "bad arguments to fibattn_theta_of_alpha");
    for (int l = 0; l < L; ++l) {
        const double a = alpha[l];
        if (!(a >= 0.5 && a <= 1.5)) return fail(FIBATTN_ERR_INVALID_ARG, "alpha[%d] = %g is outside [0.5, 1.5]", l, a);
        // theta = logit(alpha - 0.5); the ends (theta = -/+ infinity) clamp to -/+ 30
        const double t = (a <= 0.5) ? -30.0 : (a >= 1.5) ? 30.0 : std::log((a - 0.5) / (1.5 - a));
        theta[l] = (float)std::min(30.0, std::max(-30.0, t));
    }
    return FIBATTN_OK;
}

size_t fibattn_fwd_workspace_bytes(int B, int H, int T, int D, int W, int K, int dtype, const fibattn_opts* opts) {
    Resolved o;
    if (check_shape(B, H, T, D, W, K, dtype) || resolve_opts(opts, H, D, &o)) return 0;
    if (o.rotated_k) return 0;                   // the rotated keys go to the caller's buffer
    return align256((size_t)B * o.Hkv * T * kHeadDim * rot_size(dtype));
}

int fibattn_fwd(const void* q, const void* k, const void* v, void* out, float* lse,
                int B, int H, int T, int D, int W, float alpha, const float* offsets, int K,
                int dtype, const fibattn_opts* opts, void* workspace, size_t workspace_bytes, void* stream) {
    int rc = check_shape(B, H, T, D, W, K, dtype);
    if (rc) return rc;
    Resolved o;
    if ((rc = resolve_opts(opts, H, D, &o))) return rc;
    FwdArgs a;
    std::memset(&a, 0, sizeof(a));
    if ((rc = prep_rungs(alpha, offsets, K, W, o.dedup, T, &a.r, o.round_offsets))) return rc;
    if (B == 0) return FIBATTN_OK;
    if (!q || !k || !v || !out || !lse || (!workspace && !o.rotated_k))
        return fail(FIBATTN_ERR_INVALID_ARG, "NULL tensor or workspace pointer");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out) || !aligned16(lse) || !aligned16(workspace))
        return fail(FIBATTN_ERR_INVALID_ARG, "tensor pointers must be 16-byte aligned");
    size_t need = fibattn_fwd_workspace_bytes(B, H, T, D, W, K, dtype, opts);
    if (workspace_bytes < need) return fail(FIBATTN_ERR_INVALID_ARG, "workspace too small: %zu < %zu", workspace_bytes, need);
    prep_rope(o.rope_base, &a.rope);
    a.s = make_shape(B, H, T, W, o);
    void* kt = o.rotated_k ? o.rotated_k : workspace;
    a.q = q; a.k = k; a.v = v; a.out = out; a.lse = lse; a.kt = kt;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const bool bf16 = dtype == FIBATTN_BF16;
    // bf16 I/O: the tensor-core kernel when its layout applies (W <= 16,
    // K <= 16, shared memory fits), else the row-gather kernel (also the fp32
    // I/O path).
    const size_t smem_limit = 227 * 1024;
    MmaLayout ML;
    const bool mma_ok = bf16 && (o.fwd_kernel == 0 || o.fwd_kernel == 3) &&
                        build_mma_layout(a.s, a.r, o.rope_base, smem_limit - fwd_mma_static_smem(), &ML);
    if (o.fwd_kernel == 2) return fail(FIBATTN_ERR_UNSUPPORTED, "fwd_kernel 2 is not built");
    if (o.fwd_kernel == 3 && !mma_ok)
        return fail(FIBATTN_ERR_UNSUPPORTED, "requested forward kernel does not apply to these arguments "
                                             "(bf16 I/O, W <= 16, K <= 16, shared-memory layout)");
    if (o.residuals) {
        if (!mma_ok)
            return fail(FIBATTN_ERR_UNSUPPORTED, "forward residuals need the tensor-core forward (bf16 I/O, "
                                                 "fwd_kernel 0 or 3, W <= 16, K <= 16, shared-memory layout)");
        const ResLayout R = res_layout(B, H, T, W, K);
        char* rb = reinterpret_cast<char*>(o.residuals);
        a.res_qt = rb + R.qt;
        a.res_P = reinterpret_cast<float*>(rb + R.P);
        a.res_sd = reinterpret_cast<float*>(rb + R.sd);
        a.res_il = reinterpret_cast<float*>(rb + R.il);
    }
    a.S = W + 1 + K;
    if ((rc = bind_context())) return rc;
    if ((rc = status_word(&a.status))) return rc;
    cudaError_t e;
    {
        ProfScope p("rope_k", st);
        e = launch_rope_rows(k, kt, (long long)B * o.Hkv * T, T, a.rope, bf16, st, a.status);
    }
    if (e != cudaSuccess) return cuda_fail(e, "rope prologue launch");
    if (mma_ok) {
        ProfScope p("fwd", st);
        e = launch_fwd_mma(a, ML, st);
    } else {
        ProfScope p("fwd", st);
        e = launch_fwd_simple(a, bf16, st);
    }
    if (e != cudaSuccess) return cuda_fail(e, "forward launch");
    return FIBATTN_OK;
}

size_t fibattn_bwd_workspace_bytes(int B, int H, int T, int D, int W, int K, int dtype, const fibattn_opts* opts) {
    Resolved o;
    if (check_shape(B, H, T, D, W, K, dtype) || resolve_opts(opts, H, D, &o)) return 0;
    return bwd_layout(B, H, o.Hkv, T, W, K, dtype, !o.rotated_k).total;
}

int fibattn_bwd(const void* q, const void* k, const void* v, const void* out, const float* lse, const void* dout,
                void* dq, void* dk, void* dv, float* dtheta, float* dd,
                int B, int H, int T, int D, int W, float alpha, const float* offsets, int K,
                int dtype, const fibattn_opts* opts, void* workspace, size_t workspace_bytes, void* stream) {
    int rc = check_shape(B, H, T, D, W, K, dtype);
    if (rc) return rc;
    Resolved o;
    if ((rc = resolve_opts(opts, H, D, &o))) return rc;
    BwdArgs a;
    std::memset(&a, 0, sizeof(a));
    if ((rc = prep_rungs(alpha, offsets, K, W, o.dedup, T, &a.r, o.round_offsets))) return rc;
    if (o.round_offsets && (dtheta || dd))
        return fail(FIBATTN_ERR_INVALID_ARG, "rounded rung distances do not vary with alpha: pass dtheta = dd = NULL");
    if (!workspace) return fail(FIBATTN_ERR_INVALID_ARG, "workspace is NULL");
    if (B > 0 && (!q || (!k && !o.rotated_k) || !v || !lse || !dout || !dq || !dk || !dv))
        return fail(FIBATTN_ERR_INVALID_ARG, "NULL tensor pointer");
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(lse) || !aligned16(dout) || !aligned16(dq) ||
        !aligned16(dk) || !aligned16(dv) || !aligned16(workspace) || !aligned16(out) || ((uintptr_t)dtheta & 3u) ||
        ((uintptr_t)dd & 3u))
        return fail(FIBATTN_ERR_INVALID_ARG, "pointers must be 16-byte aligned (dtheta, dd: 4-byte)");
    BwdLayout L = bwd_layout(B, H, o.Hkv, T, W, K, dtype, !o.rotated_k);
    if (workspace_bytes < L.total) return fail(FIBATTN_ERR_INVALID_ARG, "workspace too small: %zu < %zu", workspace_bytes, L.total);
    prep_rope(o.rope_base, &a.rope);
    a.s = make_shape(B, H, T, W, o);
    char* ws = reinterpret_cast<char*>(workspace);
    a.q = q; a.k = k; a.v = v; a.out = out; a.lse = lse; a.dout = dout; a.dq = dq; a.dk = dk; a.dv = dv;
    a.dtheta = dtheta; a.dd = dd;
    a.want_dd = (dtheta || dd) ? 1 : 0;
    a.qt = ws + L.qt; a.kt = o.rotated_k ? o.rotated_k : ws + L.kt;
    a.P = reinterpret_cast<float*>(ws + L.P); a.DP = reinterpret_cast<float*>(ws + L.DP);
    a.Delta = reinterpret_cast<float*>(ws + L.Delta);
    a.rpart = reinterpret_cast<long long*>(ws + L.rpart);
    a.nblk_q = bwd_simple_blocks(a.s);
    a.S = W + 1 + K;
    a.alpha = alpha;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const bool bf16 = dtype == FIBATTN_BF16;
    MmaLayout ML, KL;
    const size_t smem_limit = 227 * 1024 - bwd_mma_static_smem();
    const bool mma_ok = bf16 && out && (o.bwd_kernel == 0 || o.bwd_kernel == 2) &&
                        build_mma_layout(a.s, a.r, o.rope_base, smem_limit, &ML, 3 * kTileRows) &&
                        build_key_layout(a.s, a.r, o.rope_base, 227 * 1024 - bwd_key_mma_static_smem(), &KL);
    a.Ps = reinterpret_cast<float*>(ws + L.P);      // slot-major p and dS of the tensor-core passes
    a.DSs = reinterpret_cast<float*>(ws + L.DP);
    if (o.bwd_kernel == 2 && !mma_ok)
        return fail(FIBATTN_ERR_UNSUPPORTED, "tensor-core backward needs bf16, out, W <= 16, K <= 16 and a staged row "
                                             "union that fits shared memory");
    if (mma_ok) a.nblk_q = bwd_mma_blocks(a.s);
    if (mma_ok && o.residuals &&                 // p, sd and q~ from the forward
        bwd_key_mma_smem_bytes(KL, true) + bwd_key_mma_static_smem() <= 227 * 1024) {
        const ResLayout R = res_layout(B, H, T, W, K);
        char* rb = reinterpret_cast<char*>(o.residuals);
        a.saved = 1;
        a.qt = rb + R.qt;
        a.Ps = reinterpret_cast<float*>(rb + R.P);
        a.res_sd = reinterpret_cast<const float*>(rb + R.sd);
        a.res_il = reinterpret_cast<const float*>(rb + R.il);
    }
    cudaError_t e;
    if ((rc = bind_context())) return rc;
    if ((rc = status_word(&a.status))) return rc;
    if (B > 0) {
        if (!mma_ok) {
            ProfScope p("rope_q", st);
            e = launch_rope_rows(q, a.qt, (long long)B * H * T, T, a.rope, bf16, st, a.status);
            if (e != cudaSuccess) return cuda_fail(e, "rope prologue (q) launch");
        }
        if (!o.rotated_k) {                      // else the rotated keys come from the forward
            ProfScope p("rope_k", st);
            e = launch_rope_rows(k, a.kt, (long long)B * o.Hkv * T, T, a.rope, bf16, st, a.status);
            if (e != cudaSuccess) return cuda_fail(e, "rope prologue (k) launch");
        }
        if (mma_ok) {
            ProfScope p("bwd_query_mma", st);
            e = launch_bwd_query_mma(a, ML, st);
        } else {
            ProfScope p("bwd_query", st);
            e = launch_bwd_query(a, bf16, st);
        }
        if (e != cudaSuccess) return cuda_fail(e, "backward query-pass launch");
        if (mma_ok) {
            ProfScope p("bwd_key_mma", st);
            e = launch_bwd_key_mma(a, KL, st);
        } else {
            ProfScope p("bwd_key", st);
            e = launch_bwd_key(a, bf16, st);
        }
        if (e != cudaSuccess) return cuda_fail(e, "backward key-pass launch");
    }
    if (B == 0) {                                // no queries: every gradient is zero
        e = dtheta ? cudaMemsetAsync(dtheta, 0, sizeof(float), st) : cudaSuccess;
        if (e == cudaSuccess && dd && K > 0) e = cudaMemsetAsync(dd, 0, sizeof(float) * K, st);
        if (e != cudaSuccess) return cuda_fail(e, "zero gradients for an empty batch");
        return FIBATTN_OK;
    }
    return FIBATTN_OK;                           // dtheta and dd: written by block 0 of the key pass
}

int fibattn_check_status(void* stream, unsigned* flags) {
    if (flags) *flags = 0u;
    int rc = bind_context();
    if (rc) return rc;
    unsigned* word = nullptr;
    if ((rc = status_word(&word))) return rc;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    unsigned h = 0u;
    cudaError_t e = cudaMemcpyAsync(&h, word, sizeof(h), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e == cudaSuccess && h) e = cudaMemsetAsync(word, 0, sizeof(unsigned), st);
    if (e == cudaSuccess && h) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "reading the device status word");
    if (flags) *flags = h;
    if (h & kStatusWaitTimeout)
        return fail(FIBATTN_ERR_INTERNAL, "a kernel gave up waiting for a staging copy (outputs of the affected "
                                          "tiles are NaN)%s", (h & kStatusRange) ? "; a rotated q or k row also "
                                          "overflowed fp16" : "");
    if (h & kStatusRange)
        return fail(FIBATTN_ERR_RANGE, "a RoPE-rotated q or k entry reached 65520 in magnitude, beyond the fp16 "
                                       "rows of the bf16 path (scores with such operands are not meaningful)");
    return FIBATTN_OK;
}

int fibattn_test_wait_timeout(unsigned timeout_us, void* stream) {
    if (timeout_us == 0u || timeout_us > 10000000u)
        return fail(FIBATTN_ERR_INVALID_ARG, "timeout_us must be in [1, 1e7]");
    int rc = bind_context();
    if (rc) return rc;
    unsigned* word = nullptr;
    if ((rc = status_word(&word))) return rc;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    wait_timeout_probe_kernel<<<1, 32, 0, st>>>(word, (unsigned long long)timeout_us * 1000ull);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? FIBATTN_OK : cuda_fail(e, "wait-timeout probe launch");
}

int fibattn_staging_layout(int kind, int T, int W, float alpha, const float* offsets, int K, int no_dedup,
                           int* n_iv, int* iv_start, int* iv_len, int* iv_smem, int* slab_row) {
    if (kind != 0 && kind != 1) return fail(FIBATTN_ERR_INVALID_ARG, "kind must be 0 or 1");
    if (T < 1 || T > (1 << 20)) return fail(FIBATTN_ERR_INVALID_ARG, "T must be in [1, 2^20]");
    if (W < 0 || W > kMaxWindow || K < 0 || K > kMaxRungs)
        return fail(FIBATTN_ERR_INVALID_ARG, "need 0 <= W <= %d and 0 <= K <= %d", kMaxWindow, kMaxRungs);
    RungParams r;
    int rc = prep_rungs(alpha, offsets, K, W, no_dedup ? 0 : 1, T, &r);
    if (rc) return rc;
    Shape s;
    std::memset(&s, 0, sizeof(s));
    s.B = 1; s.H = 1; s.Hkv = 1; s.G = 1; s.T = T; s.W = W;
    MmaLayout L;
    std::memset(&L, 0, sizeof(L));
    const size_t no_limit = ~(size_t)0;
    const bool ok = kind == 0 ? build_mma_layout(s, r, 1e4, no_limit, &L) : build_key_layout(s, r, 1e4, no_limit, &L);
    if (!ok) return fail(FIBATTN_ERR_UNSUPPORTED, "the tensor-core layout needs W <= 16 and K <= %d", kMmaMaxRungs);
    if (n_iv) *n_iv = L.n_iv;
    for (int i = 0; i < L.n_iv; ++i) {
        if (iv_start) iv_start[i] = L.iv_start[i];
        if (iv_len) iv_len[i] = L.iv_len[i];
        if (iv_smem) iv_smem[i] = L.iv_smem[i];
    }
    for (int k = 0; k < K && slab_row; ++k) slab_row[k] = ((r.active >> k) & 1u) ? L.rung_smem[k] : -1;
    return FIBATTN_OK;
}

int fibattn_coverage(int L, const float* alphas, const float* offsets, int K, int W, int T, int no_dedup,
                     int* per_layer, int* union_count, int* beyond_window, int* two_hop) {
    if (L < 1 || L > 4096 || !alphas) return fail(FIBATTN_ERR_INVALID_ARG, "need 1 <= L <= 4096 alphas");
    if (T < 1 || T > (1 << 20)) return fail(FIBATTN_ERR_INVALID_ARG, "T must be in [1, 2^20]");
    if (W < 0 || K < 0 || K > kMaxRungs) return fail(FIBATTN_ERR_INVALID_ARG, "need W >= 0 and 0 <= K <= %d", kMaxRungs);
    std::vector<std::vector<int>> D(L);
    std::vector<char> uni(T, 0);
    for (int l = 0; l < L; ++l) {
        RungParams r;
        int rc = prep_rungs(alphas[l], offsets, K, W, no_dedup ? 0 : 1, T, &r);
        if (rc) return rc;
        std::vector<char> in(T, 0);
        for (int t = 0; t <= W && t < T; ++t) in[t] = 1;
        for (int k = 0; k < K; ++k) {
            if (!((r.active >> k) & 1u)) continue;
            if (r.s0[k] < T) in[r.s0[k]] = 1;
            if (r.w[k] != 0.f && r.s0[k] + 1 < T) in[r.s0[k] + 1] = 1;
        }
        for (int t = 0; t < T; ++t)
            if (in[t]) { D[l].push_back(t); uni[t] = 1; }
        if (per_layer) per_layer[l] = (int)D[l].size();
    }
    int u = 0, beyond = 0;
    for (int t = 0; t < T; ++t)
        if (uni[t]) { ++u; if (t > W) ++beyond; }
    if (union_count) *union_count = u;
    if (beyond_window) *beyond_window = beyond;
    if (two_hop) {
        std::vector<char> hop(T, 0);
        for (int l = 0; l + 1 < L; ++l)
            for (int a : D[l])
                for (int b : D[l + 1])
                    if (a + b < T) hop[a + b] = 1;
        int n = 0;
        for (int t = 0; t < T; ++t) n += hop[t];
        *two_hop = n;
    }
    return FIBATTN_OK;
}

}  // extern "C"
