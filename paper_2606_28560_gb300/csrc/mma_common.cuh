// mma_common.cuh -- device helpers shared by the tensor-core kernels: PTX
// wrappers (mbarrier, TMA, ldmatrix, mma.sync), fragment packing, the 128-byte
// swizzled row addressing of staged rows, and the copy issue of a staged
// row union.
#pragma once
#include <cuda.h>
#include <cudaTypedefs.h>

#include "fibattn_internal.cuh"
#include "fwd_mma.cuh"

namespace fibattn {
namespace mma {

// A wait on a staging copy gives up after this long (the copies are of at
// most a few hundred KB from L2 or HBM and land within microseconds).
constexpr unsigned long long kWaitLimitNs = 1000000000ull;   // 1 s

__device__ __forceinline__ unsigned smem_u32(const void* p) { return (unsigned)__cvta_generic_to_shared(p); }

// 4-byte asynchronous copy global -> shared; zero-filled when !full.
__device__ __forceinline__ void cp_async4(const float* dst, const float* src, bool full) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n"
                 :: "r"(smem_u32(dst)), "l"(src), "r"(full ? 4 : 0) : "memory");
}

__device__ __forceinline__ void mbar_init(unsigned long long* bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" :: "r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(unsigned long long* bar, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" :: "r"(smem_u32(bar)), "r"(bytes));
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;\n" : "=l"(t));
    return t;
}

// Bounded wait on phase `parity`: false once limit_ns of the global timer
// have passed since the first poll that did not find the phase complete (the
// timer is read every 64 polls).  The caller poisons its outputs and raises
// kStatusWaitTimeout; nothing hangs.
__device__ __forceinline__ bool mbar_wait(unsigned long long* bar, unsigned parity,
                                          unsigned long long limit_ns = kWaitLimitNs) {
    const unsigned a = smem_u32(bar);
    unsigned long long t0 = 0;
    for (unsigned it = 0;; ++it) {
        unsigned done;
        asm volatile("{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
                     " selp.u32 %0, 1, 0, p;\n}\n" : "=r"(done) : "r"(a), "r"(parity) : "memory");
        if (done) return true;
        if ((it & 63u) == 0u) {
            const unsigned long long now = global_ns();
            if (it == 0) t0 = now;
            else if (now - t0 > limit_ns) return false;
        }
    }
}
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int x, int y, int z,
                                            unsigned long long* bar) {
    asm volatile("cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
                 " [%0], [%1, {%2, %3, %4}], [%5];\n"
                 :: "r"(smem_u32(dst)), "l"(map), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void ldsm_x4(unsigned addr, unsigned& r0, unsigned& r1, unsigned& r2, unsigned& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(unsigned addr, unsigned& r0, unsigned& r1, unsigned& r2, unsigned& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3) : "r"(addr));
}

__device__ __forceinline__ void mma_f16_16816(float* d, const unsigned* a, unsigned b0, unsigned b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};\n"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// The same product into a fresh accumulator (C = 0).
__device__ __forceinline__ void mma_f16_16816_z(float* d, const unsigned* a, unsigned b0, unsigned b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%10,%10,%10,%10};\n"
                 : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(0.f));
}
__device__ __forceinline__ void mma_bf16_16816(float* d, const unsigned* a, unsigned b0, unsigned b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};\n"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma_bf16_16816_z(float* d, const unsigned* a, unsigned b0, unsigned b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%10,%10,%10,%10};\n"
                 : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1), "f"(0.f));
}
__device__ __forceinline__ void mma_bf16_1688(float* d, unsigned a0, unsigned a1, unsigned b0) {
    asm volatile("mma.sync.aligned.m16n8k8.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5}, {%6}, "
                 "{%0,%1,%2,%3};\n"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3]) : "r"(a0), "r"(a1), "r"(b0));
}

__device__ __forceinline__ unsigned pack_f16(float lo, float hi) {
    __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<unsigned*>(&h);
}
__device__ __forceinline__ unsigned pack_bf16(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<unsigned*>(&h);
}

// Two bf16 ones: a B fragment of all ones makes an MMA return the row sums
// of its A operand (exactly the rounded entries the value product uses).
constexpr unsigned kOnesBf16x2 = 0x3f803f80u;

// 2^x by the hardware approximation (MUFU); x = -inf gives +0.
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;\n" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float quad_sum(float x) {
    x += __shfl_xor_sync(0xffffffffu, x, 1);
    x += __shfl_xor_sync(0xffffffffu, x, 2);
    return x;
}
__device__ __forceinline__ float quad_max(float x) {
    x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 1));
    x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, 2));
    return x;
}

// Shared-memory byte address of 16-byte chunk `ch` (< 8) of staged row `row`
// under the 128-byte swizzle (chunk index XOR row % 8), buffer base 1024-byte
// aligned.  XOR being linear, chunk ch ^ m of the same row is at the address
// XOR (m << 4), and the row 8 further on 1024 bytes on.
__device__ __forceinline__ unsigned row_chunk(unsigned base, int row, int ch) {
    return base + ((unsigned)row << 7) + ((unsigned)((row ^ ch) & 7) << 4);
}

// Warp 0 issues the copies of one staged tensor.  Lane n copies merged
// interval n: whole 64-row boxes (map64) first, then 8-row boxes (map8) for
// the rest of it (interval lengths are multiples of 8 rows).  Large boxes move
// the same rows at well over the rate of 8-row ones.  Lane 0 announces the
// byte count before any copy is issued.
__device__ __forceinline__ void issue_rows(unsigned char* dst, const CUtensorMap* map64, const CUtensorMap* map8,
                                           const MmaLayout& L, int i0, int head, unsigned long long* bar, int lane) {
    if (lane == 0) mbar_expect_tx(bar, (unsigned)L.rows * 128u);
    __syncwarp();
    for (int iv = lane; iv < L.n_iv; iv += 32) {
        const int len = L.iv_len[iv], srow = L.iv_smem[iv], grow = i0 + L.iv_start[iv];
        int r = 0;
        for (; r + 64 <= len; r += 64) tma_load_3d(dst + (size_t)(srow + r) * 128, map64, 0, grow + r, head, bar);
        for (; r < len; r += 8) tma_load_3d(dst + (size_t)(srow + r) * 128, map8, 0, grow + r, head, bar);
    }
}

// One batch of the copies issue_rows makes: boxes that start at or after
// L.lo_start (hi_batch false) or before it (hi_batch true); the barrier
// expects that batch's bytes.  Boxes are the same as issue_rows's.
__device__ __forceinline__ void issue_rows_batch(unsigned char* dst, const CUtensorMap* map64, const CUtensorMap* map8,
                                                 const MmaLayout& L, int i0, int head, unsigned long long* bar,
                                                 int lane, bool hi_batch) {
    if (lane == 0) mbar_expect_tx(bar, hi_batch ? L.bytes_hi : L.bytes_lo);
    __syncwarp();
    for (int iv = lane; iv < L.n_iv; iv += 32) {
        const int len = L.iv_len[iv], srow = L.iv_smem[iv], grow = i0 + L.iv_start[iv];
        int r = 0;
        for (; r + 64 <= len; r += 64)
            if ((srow + r < L.lo_start) == hi_batch) tma_load_3d(dst + (size_t)(srow + r) * 128, map64, 0, grow + r, head, bar);
        for (; r < len; r += 8)
            if ((srow + r < L.lo_start) == hi_batch) tma_load_3d(dst + (size_t)(srow + r) * 128, map8, 0, grow + r, head, bar);
    }
}

// One thread copies merged interval iv (64-row boxes, then 8-row boxes) under
// barrier `bar`, which it arms with the interval's byte count first.
__device__ __forceinline__ void issue_interval(unsigned char* dst, const CUtensorMap* map64, const CUtensorMap* map8,
                                               const MmaLayout& L, int iv, int i0, int head, unsigned long long* bar) {
    const int len = L.iv_len[iv], srow = L.iv_smem[iv], grow = i0 + L.iv_start[iv];
    mbar_expect_tx(bar, (unsigned)len * 128u);
    int r = 0;
    for (; r + 64 <= len; r += 64) tma_load_3d(dst + (size_t)(srow + r) * 128, map64, 0, grow + r, head, bar);
    for (; r < len; r += 8) tma_load_3d(dst + (size_t)(srow + r) * 128, map8, 0, grow + r, head, bar);
}

// The RoPE phase steps of the 32 pairs (see RopeParams) and the cos, sin of 8
// position steps, copied into shared memory once per CTA: a thread reads the
// pairs of its fragment columns, which differ between the lanes of a warp, and
// lane-dependent reads of kernel parameters are serialised.
struct RopeSmem {
    unsigned long long F[kHalf];
    float c8[kHalf], s8[kHalf];
};
// Called by threads 0..31 (or all: others do nothing) before a CTA barrier.
__device__ __forceinline__ void rope_to_smem(RopeSmem& r, const RopeParams& rp, const MmaLayout& L, int tid) {
    if (tid < kHalf) {
        r.F[tid] = rp.F[tid];
        r.c8[tid] = L.rope_c8[tid];
        r.s8[tid] = L.rope_s8[tid];
    }
}
// cos/sin of the angle of pair m at position pos (as rope_cs).
__device__ __forceinline__ void rope_cs_s(const RopeSmem& r, int m, int pos, float& c, float& s) {
    const unsigned long long ph = (unsigned long long)(unsigned)pos * r.F[m];
    const int hi = (int)(unsigned)(ph >> 32);        // signed turn fraction in [-1/2, 1/2)
    __sincosf((float)hi * 1.4629180792671596e-09f, &s, &c);   // 2*pi / 2^32
}

// Shared-memory counter increment with acquire-release order (CTA scope);
// returns the old value.
__device__ __forceinline__ unsigned atom_add_acq_rel(unsigned* p, unsigned v) {
    unsigned old;
    asm volatile("atom.acq_rel.cta.shared::cta.add.u32 %0, [%1], %2;\n" : "=r"(old) : "r"(smem_u32(p)), "r"(v)
                 : "memory");
    return old;
}

__device__ __forceinline__ void mma_f16_1688(float* d, unsigned a0, unsigned a1, unsigned b0) {
    asm volatile("mma.sync.aligned.m16n8k8.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5}, {%6}, "
                 "{%0,%1,%2,%3};\n"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3]) : "r"(a0), "r"(a1), "r"(b0));
}

}  // namespace mma
}  // namespace fibattn
