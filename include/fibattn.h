/*
 * fibattn.h -- C ABI of the GB300 (sm_103a) library for depth-staggered
 * scaled-Fibonacci sparse attention (arXiv 2606.28560).
 *
 * The operation (Section 2, "Attended set"): query i attends to the dense
 * causal window at distances 0..W plus K rungs at continuous distances
 * d_k = alpha * f_k.  A rung is read by linear interpolation between the
 * floor and floor-plus-one positions; RoPE is applied to q and k at their true
 * positions before the gather; the attended scores go through a softmax and
 * weight the (equally interpolated) values.  alpha = 0.5 + sigmoid(theta) is
 * one scalar per layer (Section 2, "The per-layer scalar").
 *
 * Conventions shared by every call:
 *   - Tensor layouts are row-major and contiguous: q, out, dout, dq are
 *     [B][H][T][D]; k, v, dk, dv are [B][Hkv][T][D]; lse is [B][H][T] fp32.
 *     Element type is given by `dtype` (fp32 or bf16); lse is always fp32.
 *   - Tensor, workspace and output-scalar pointers are DEVICE pointers owned by
 *     the caller and aligned to 16 bytes.  `offsets` is a HOST array of K floats
 *     (the base sequence f_k, e.g. 1,2,3,5,...,987) read during the call only.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Device work is asynchronous on that stream; a call returns after launch.
 *     Work goes to the calling thread's current device; a compute call makes
 *     that device's primary context current on the thread if none is.
 *   - Return value is a fibattn_status.  Argument errors are reported before
 *     any launch.  Faults raised asynchronously by the device surface at the
 *     caller's next synchronisation.  fibattn_last_error() gives a thread-local
 *     message for the last non-OK status.  No C++ exception crosses the ABI.
 *   - Limits: D == 64; 0 <= W <= 1024; 0 <= K <= 32; 1 <= T <= 2^20;
 *     0.5 <= alpha <= 1.5; every d_k = fl32(alpha * f_k) must be finite and
 *     >= 0; H % Hkv == 0.
 *   - Readings of the paper taken where it is silent: scale = 1/sqrt(D); the
 *     floor is taken of the distance, the far row i-floor(d)-1 has weight
 *     d-floor(d); a rung with d_k > i is masked; with dedup a rung with
 *     d_k <= W is dropped (the attended set is a set union); RoPE pairs
 *     dimension m with m+D/2 at frequency rope_base^(-2m/D).
 */
#ifndef FIBATTN_H
#define FIBATTN_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    FIBATTN_OK = 0,
    FIBATTN_ERR_INVALID_ARG = 1,   /* bad shape, pointer, alignment, alpha, ...   */
    FIBATTN_ERR_UNSUPPORTED = 2,   /* valid but not built (e.g. D != 64)           */
    FIBATTN_ERR_CUDA = 3,          /* a CUDA runtime call or launch failed         */
    FIBATTN_ERR_INTERNAL = 4,      /* an internal consistency check failed, or a
                                      kernel gave up a bounded wait (see
                                      fibattn_check_status)                        */
    FIBATTN_ERR_RANGE = 5          /* an operand left the range of the library's
                                      16-bit rotated rows (fibattn_check_status)   */
} fibattn_status;

typedef enum { FIBATTN_F32 = 0, FIBATTN_BF16 = 1 } fibattn_dtype;

/* Options.  Zero-initialised fields take the defaults in brackets. */
typedef struct {
    float rope_base;   /* RoPE frequency base [1e4] (Section 3, "Model and training") */
    float scale;       /* score scale; <= 0 means 1/sqrt(D)                            */
    int   Hkv;         /* key/value heads (GQA); 0 means Hkv = H                       */
    int   no_dedup;    /* 0: drop rungs with d_k <= W [default]; 1: keep them          */
    int   fwd_kernel;  /* forward kernel: 0 automatic [default]; 1 row-gather kernel
                          (any W and K, fp32 or bf16); 3 tensor-core kernel (bf16
                          I/O, W <= 16, K <= 16); 2 is not built.
                          FIBATTN_ERR_UNSUPPORTED when the choice does not apply. */
    int   bwd_kernel;  /* backward query pass: 0 automatic [default]; 1 row-gather
                          single sweep (Delta accumulated from the slots, `out`
                          unused); 2 tensor-core kernel (bf16 I/O, `out` given,
                          W <= 16, K <= 16; FIBATTN_ERR_UNSUPPORTED otherwise).
                          Automatic takes 2 where it applies, else 1. */
    void* rotated_k;   /* optional device buffer of B*Hkv*T*D elements (fp16 for bf16
                          I/O, fp32 for fp32 I/O), 16-byte aligned [NULL].  Given
                          it, fibattn_fwd writes the RoPE-rotated keys there
                          instead of into its workspace, and fibattn_bwd reads
                          them from there instead of rotating k again (k may then
                          be NULL): a caller that keeps this buffer from the
                          forward to the backward keeps it in place of k. */
    void* residuals;   /* optional device buffer of fibattn_residual_bytes(...) bytes,
                          16-byte aligned [NULL].  Given it, fibattn_fwd also writes
                          what the backward would otherwise recompute from q and k:
                          the RoPE-rotated queries (bf16 [B][H][T][D]), the
                          unnormalised softmax weight exp(s - max) of every
                          slot (fp32 [B][H][S][T], S = W + 1 + K: window
                          distances 0..W, then rung k at W + 1 + k; 0 where not
                          attended; rungs that are never read -- dropped by
                          dedup or beyond T's reach -- are left unwritten), the
                          far-minus-floor raw score q~ . (k~_far - k~_floor) of
                          every rung (fp32 [B][H][K][T]) and 1 / (sum of the
                          weights) per query (fp32 [B][H][T]), so that the
                          probability is weight / sum; the four arrays follow
                          one another in
                          that order, each starting at the next multiple of 256
                          bytes.  Only the tensor-core forward writes them:
                          bf16 I/O, and fwd_kernel 0 or 3 with its layout applying;
                          otherwise fibattn_fwd fails with FIBATTN_ERR_UNSUPPORTED
                          before any launch.  fibattn_bwd given the buffer filled by
                          the forward of the same inputs and parameters reads them
                          in its tensor-core passes instead of recomputing the
                          scores; when its tensor-core passes do not apply it
                          ignores the buffer. */
    int   round_offsets; /* 0: continuous distances d_k = fl32(alpha f_k), rungs
                          interpolated [default]; 1: the integer-offset variants
                          (Section 2, "Implementation note", the fused
                          boolean-mask path): d_k rounded to the nearest integer,
                          ties to even, after the fp32 product; every rung then
                          reads one row.  fibattn_bwd then requires dtheta and dd
                          to be NULL (the rounded distances do not vary with
                          alpha). */
} fibattn_opts;

/* ---------------------------------------------------------------------------
 * Forward: out[b,h,i,:] and lse[b,h,i] (log of the softmax normaliser, in the
 * scaled-score domain) for every query (Section 2, "Attended set").
 * workspace: device scratch of at least fibattn_fwd_workspace_bytes(...)
 * bytes; contents on entry are ignored and on exit are unspecified.
 * out may not alias q, k, v or workspace.
 * ------------------------------------------------------------------------- */
size_t fibattn_fwd_workspace_bytes(int B, int H, int T, int D, int W, int K,
                                   int dtype, const fibattn_opts* opts);

int fibattn_fwd(const void* q, const void* k, const void* v,
                void* out, float* lse,
                int B, int H, int T, int D, int W,
                float alpha, const float* offsets, int K,
                int dtype, const fibattn_opts* opts,
                void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * Backward (the chain rule of the forward definition; the paper trains every
 * model through this path, Section 2 "Implementation note").
 * Inputs: q, k, v, dout as above and lse from fibattn_fwd of the same inputs.
 * out: the output of that forward call, or NULL.  With out, the softmax term
 * Delta_i = sum_slots p dp (= dout_i . out_i) is read as dout_i . out_i, which
 * lets the tensor-core query pass (opts->bwd_kernel) form each score gradient
 * in one pass; without it Delta is accumulated from the slots.
 * Outputs (overwritten, not accumulated): dq [B,H,T,D], dk and dv [B,Hkv,T,D]
 * in `dtype`, gradients with respect to the pre-RoPE q and k; dtheta (device,
 * 1 float, may be NULL) = dL/dtheta with alpha = 0.5 + sigmoid(theta); dd
 * (device, K floats, may be NULL) = dL/dd_k for each rung distance.
 * dL/dalpha = sum_k f_k dd_k.  With both NULL (a fixed alpha schedule, alpha
 * not trained) the rung-distance gradient is not computed at all.
 * At an integer d_k the distance derivative is one-sided, from above.
 * dq, dk, dv, dtheta and dd may not alias each other, an input, the
 * residuals or the workspace.
 * ------------------------------------------------------------------------- */
size_t fibattn_bwd_workspace_bytes(int B, int H, int T, int D, int W, int K,
                                   int dtype, const fibattn_opts* opts);

int fibattn_bwd(const void* q, const void* k, const void* v,
                const void* out, const float* lse, const void* dout,
                void* dq, void* dk, void* dv, float* dtheta, float* dd,
                int B, int H, int T, int D, int W,
                float alpha, const float* offsets, int K,
                int dtype, const fibattn_opts* opts,
                void* workspace, size_t workspace_bytes, void* stream);

/* Bytes of the forward residuals (fibattn_opts.residuals) for these sizes;
 * 0 for invalid sizes or fp32 I/O (no residuals). */
size_t fibattn_residual_bytes(int B, int H, int T, int D, int W, int K, int dtype);

/* Thread-local message for the last non-OK status returned on this thread. */
const char* fibattn_last_error(void);

/* ---------------------------------------------------------------------------
 * Device status (no counterpart in the paper).  Kernels report two conditions
 * that no argument check can catch before launch into a per-device status
 * word, without stopping:
 *   bit 0 -- a kernel gave up waiting for one of its own shared-memory staging
 *            copies (each wait is bounded to 1 s of the GPU's global timer);
 *            the affected tiles' outputs (out, lse, gradients) are NaN.
 *   bit 1 -- an entry of a 16-bit rotated row reached 65520 in magnitude:
 *            the bf16 path keeps the RoPE-rotated keys, and the rotated
 *            queries times the score scale, in fp16 (for score precision),
 *            which cannot hold it.
 * fibattn_check_status synchronises `stream`, reads the calling thread's
 * current device's word into *flags (may be NULL) and clears it.  Returns
 * FIBATTN_ERR_INTERNAL if bit 0 was set, else FIBATTN_ERR_RANGE if bit 1 was
 * set, else FIBATTN_OK.  Compute calls never synchronise to look at it.
 * ------------------------------------------------------------------------- */
int fibattn_check_status(void* stream, unsigned* flags);

/* Test hook for the bounded wait: launches one warp on `stream` that waits on
 * a shared-memory barrier no copy will complete, with a bound of timeout_us
 * microseconds (1 .. 1e7); the wait runs out and sets status bit 0, which a
 * following fibattn_check_status reports.  The kernel touches no memory but
 * its own shared barrier and the status word. */
int fibattn_test_wait_timeout(unsigned timeout_us, void* stream);

/* ---------------------------------------------------------------------------
 * Host-side parameter prep (no GPU needed).
 * ------------------------------------------------------------------------- */

/* Rung prep (Section 2): d[k] = fl32(alpha * f[k]) (with round_offsets then
 * rounded to the nearest integer, ties to even); s0[k] = floor(d[k]);
 * w[k] = d[k] - s0[k]; active[k] = 1 unless dedup drops it (d[k] <= W).
 * Any output pointer may be NULL.  Host pointers. */
int fibattn_rung_params(float alpha, const float* offsets, int K, int W, int no_dedup, int round_offsets,
                        float* d, int* s0, float* w, int* active);

/* Base sequences (Section 2): kind 0 = Fibonacci 1,2,3,5,... ; kind 1 =
 * powers of two 1,2,4,... .  Writes K floats to host array f. */
int fibattn_base(int kind, int K, float* f);

/* Per-layer alpha schedules (Section 2, "The per-layer scalar"):
 * kind 0 fixed (alpha = 1); 1 learned (alpha_l = 0.5 + sigmoid(theta[l]));
 * 2 linear stagger (alpha_l = 0.5 + l/(L-1)); 3 coprime reassignment of the
 * linear multiset, layer l takes linear index (stride*l mod L).
 * theta is read only for kind 1.  Host arrays. */
int fibattn_alpha_schedule(int kind, int L, const float* theta, int stride, float* alpha);

/* Inverse of the learned map on [0.5, 1.5]: theta[l] = log((alpha[l] - 0.5) /
 * (1.5 - alpha[l])), the ends (theta = -/+ infinity) clamped to -/+ 30; used to
 * start a learned theta at a static schedule's alpha.  Host arrays. */
int fibattn_theta_of_alpha(int L, const float* alpha, float* theta);

/* ---------------------------------------------------------------------------
 * Coverage of a layer stack (Section 4.2, "Why staggering widens coverage"):
 * the distinct key distances i - j a query reads.  Layer l (alpha = alphas[l])
 * reads D_l = {0..W} plus, for each active rung with d_k <= T-1 (the rung
 * prep of fibattn_rung_params, with T's reach), the floor row's distance
 * floor(d_k) and, when d_k is fractional, the far row's floor(d_k)+1.
 * Outputs (each may be NULL): per_layer[l] = |D_l| (L ints); union_count =
 * |union of D_l|; beyond_window = |union of D_l minus {0..W}|; two_hop =
 * |union over l of {a + b < T : a in D_l, b in D_l+1}| (what a query's
 * representation after two successive layers draws on).  Host arrays;
 * 1 <= L <= 4096, 1 <= T <= 1<<20.
 * ------------------------------------------------------------------------- */
int fibattn_coverage(int L, const float* alphas, const float* offsets, int K, int W, int T, int no_dedup,
                     int* per_layer, int* union_count, int* beyond_window, int* two_hop);

/* ---------------------------------------------------------------------------
 * Shared-memory staging layout of the tensor-core kernels (host-side, no GPU;
 * a diagnostic without counterpart in the paper).  A CTA of these kernels owns
 * a tile of 120 consecutive queries (kind 0: the forward and the backward
 * query pass) or keys (kind 1: the backward key pass) and stages the rows its
 * warps read: for kind 0 the window band [-Wp, 121) and, per staged rung k,
 * the slab [-s0_k - 1, 121 - s0_k) relative to the tile's first query (Wp =
 * 0, 8 or 16 for W = 0, <= 8, <= 16); for kind 1 the band [0, 121 + Wp) and
 * the slabs [s0_k, s0_k + 121) relative to the first key.  Overlapping row
 * ranges are merged and each merged interval is rounded up to whole 8-row
 * copies.  Outputs (host arrays of at least 17 ints, any may be NULL):
 * n_iv intervals with relative first row iv_start, row count iv_len and first
 * shared row iv_smem; slab_row[k] (K ints) = shared row of the first row of
 * rung k's slab, -1 when the rung is not staged (dropped by dedup or beyond
 * T's reach).  FIBATTN_ERR_UNSUPPORTED when the tensor-core kernels do not
 * apply (W > 16 or K > 16).
 * ------------------------------------------------------------------------- */
int fibattn_staging_layout(int kind, int T, int W, float alpha, const float* offsets, int K, int no_dedup,
                           int* n_iv, int* iv_start, int* iv_len, int* iv_smem, int* slab_row);

/* ---------------------------------------------------------------------------
 * Forward without a caller-provided workspace.  The paper has no counterpart;
 * this serves callers that cannot allocate device memory -- a host framework
 * that owns all device memory and gives its plugins only tensors, or a hot
 * path where cudaMalloc's implicit device synchronisation is not allowed.
 * Same arguments and results as fibattn_fwd without workspace/workspace_bytes.
 * Scratch: one library-owned device array of FIBATTN_NOALLOC_SCRATCH_BYTES
 * (32 MiB, enough for B*Hkv*T <= 262144 bf16 rows or 131072 fp32 rows), held
 * by every GPU that loads the library until the process exits.  Calls that
 * need more are rejected with FIBATTN_ERR_INVALID_ARG before any device work.
 * The call allocates nothing (no cudaMalloc / cudaFree).  The first call on
 * each device looks up the array's device address with that device current;
 * make that first call before any stream capture.  Every call shares the one
 * array and leaves its contents behind: calls that overlap on the GPU (other
 * streams, other host threads) race on it and must be serialised by the caller.
 * ------------------------------------------------------------------------- */
#define FIBATTN_NOALLOC_SCRATCH_BYTES (32u << 20)
int fibattn_fwd_noalloc(const void* q, const void* k, const void* v, void* out, float* lse,
                        int B, int H, int T, int D, int W, float alpha, const float* offsets, int K,
                        int dtype, const fibattn_opts* opts, void* stream);

/* ---------------------------------------------------------------------------
 * Opt-in kernel timing (no counterpart in the paper; used to attribute time
 * to kernels).  fibattn_profile_enable(1) clears the record and brackets every
 * later launch with CUDA events on the launch stream; (0) stops and clears.
 * Launches made while the stream is being captured into a CUDA graph record
 * external event nodes, so the summary then reports the graph's last replay.
 * fibattn_profile_summary(-1, ...) returns the number of distinct kernels
 * recorded; with index i >= 0 it synchronises on those events and writes the
 * kernel name, its summed device time in ms and its launch count.
 * ------------------------------------------------------------------------- */
int fibattn_profile_enable(int on);
int fibattn_profile_summary(int index, char* name, int name_len, double* total_ms, int* launches);

#ifdef __cplusplus
}
#endif

#endif /* FIBATTN_H */
