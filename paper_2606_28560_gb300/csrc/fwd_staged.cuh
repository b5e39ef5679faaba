// fwd_staged.cuh -- host/device interface of the staged forward kernel.
#pragma once
#include "fibattn_internal.cuh"

namespace fibattn {

constexpr int kStagedM = 128;        // queries per CTA
constexpr int kStagedR = 8;          // consecutive queries per lane group
constexpr int kMaxIntervals = kMaxRungs + 1;

// Union of the row intervals a query tile [i0, i0+M) reads, relative to i0:
// the window band [-W, M) and one slab [-s0-1, M-s0) per active rung, merged.
// Interval n covers relative rows [iv_start[n], iv_start[n] + iv_len[n]) and is
// stored from shared-memory row iv_smem[n].
struct StageLayout {
    int n_iv;
    int rows;                         // shared-memory rows in total (128 B each)
    int slot_pitch;                   // floats per query row of the score table (odd)
    int win_smem;                     // shared row of relative row 0 (window band is win_smem + rel)
    int iv_start[kMaxIntervals];
    int iv_len[kMaxIntervals];
    int iv_smem[kMaxIntervals];
    int rung_smem[kMaxRungs];         // shared row of relative row -s0_k - 1
    float rope_c1[kHalf];             // cos, sin of one position step of pair m
    float rope_s1[kHalf];
};

// Builds the layout for the rung parameters; returns false when the staged
// kernel does not apply (shared memory would exceed `smem_limit`).
bool build_stage_layout(const Shape& s, const RungParams& r, double rope_base, size_t smem_limit, StageLayout* L);
size_t fwd_staged_smem_bytes(const StageLayout& L);
cudaError_t launch_fwd_staged(const FwdArgs& a, const StageLayout& L, bool bf16, cudaStream_t st);

}  // namespace fibattn
