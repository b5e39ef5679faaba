// stage_layout.cu -- host-side layout of the rows a query tile stages in
// shared memory (see fwd_staged.cuh).
#include <algorithm>
#include <cmath>
#include <vector>

#include "fwd_staged.cuh"

namespace fibattn {

bool build_stage_layout(const Shape& s, const RungParams& r, double rope_base, size_t smem_limit, StageLayout* L) {
    const int M = kStagedM;
    struct Iv { int a, b; };                      // [a, b) relative rows
    std::vector<Iv> iv;
    iv.push_back({-s.W, M});
    for (int k = 0; k < r.K; ++k)
        if ((r.active >> k) & 1u) iv.push_back({-r.s0[k] - 1, M - r.s0[k]});
    std::sort(iv.begin(), iv.end(), [](const Iv& x, const Iv& y) { return x.a < y.a; });
    std::vector<Iv> merged;
    for (const Iv& x : iv) {
        if (!merged.empty() && x.a <= merged.back().b) merged.back().b = std::max(merged.back().b, x.b);
        else merged.push_back(x);
    }
    if ((int)merged.size() > kMaxIntervals) return false;
    L->n_iv = (int)merged.size();
    int rows = 0;
    for (int n = 0; n < L->n_iv; ++n) {
        L->iv_start[n] = merged[n].a;
        L->iv_len[n] = merged[n].b - merged[n].a;
        L->iv_smem[n] = rows;
        rows += L->iv_len[n];
    }
    L->rows = rows;
    auto smem_row = [&](int rel) {
        for (int n = 0; n < L->n_iv; ++n)
            if (rel >= L->iv_start[n] && rel < L->iv_start[n] + L->iv_len[n]) return L->iv_smem[n] + (rel - L->iv_start[n]);
        return -1;
    };
    L->win_smem = smem_row(0);
    for (int k = 0; k < kMaxRungs; ++k) L->rung_smem[k] = 0;
    for (int k = 0; k < r.K; ++k)
        if ((r.active >> k) & 1u) L->rung_smem[k] = smem_row(-r.s0[k] - 1);
    const int nslot = s.W + 1 + r.K;
    L->slot_pitch = nslot | 1;
    for (int m = 0; m < kHalf; ++m) {
        double theta = std::pow(rope_base, -2.0 * m / (double)kHeadDim);
        L->rope_c1[m] = (float)std::cos(theta);
        L->rope_s1[m] = (float)std::sin(theta);
    }
    return fwd_staged_smem_bytes(*L) <= smem_limit;
}

}  // namespace fibattn
