// fwd_mma.cuh -- host/device interface of the tensor-core forward kernel.
#pragma once
#include <cuda.h>

#include "fibattn_internal.cuh"

namespace fibattn {

constexpr int kMmaWarps = 8;                      // one 16-row MMA tile per warp
constexpr int kMmaTile = kMmaWarps * 15;          // queries per CTA (tiles every 15 rows)
constexpr int kMmaMaxRungs = 16;

// Rows a CTA stages, relative to its first query: merged intervals of the
// window band [-Wp, M+1) and the rung slabs [-s0-1, M+1-s0), each rounded up
// to whole 8-row TMA boxes and stored from shared row iv_smem[n].
struct MmaLayout {
    int n_iv;
    int rows;
    int nt;                                       // window n-tiles: 16 + Wp = 8 nt keys
    int win_smem;                                 // shared row of relative row 0
    int iv_start[kMmaMaxRungs + 1];
    int iv_len[kMmaMaxRungs + 1];
    int iv_smem[kMmaMaxRungs + 1];
    int rung_smem[kMmaMaxRungs];                  // shared row of relative row -s0_k - 1
    float rope_c8[kHalf];                         // cos, sin of 8 position steps of pair m
    float rope_s8[kHalf];
    // The active rungs in increasing d (so the rungs a tile can use form a
    // prefix); entries n_act.. pad the list with zero weight and shared row 0.
    int n_act;
    int act_k[kMmaMaxRungs];
    int act_s0[kMmaMaxRungs];
    int act_smem[kMmaMaxRungs];
    float act_w[kMmaMaxRungs];
    float act_d[kMmaMaxRungs];
    int act_iv[kMmaMaxRungs];                     // merged interval that holds the rung's slab
    int win_iv;                                   // merged interval that holds the window band
    // Staging buffer rows (>= rows).  A kernel that first copies its tile's own
    // rows (128 per tensor: q in the forward; q, dO, o in the query backward)
    // to buffer rows [0, reserved rows) issues the copy boxes that start at or
    // after lo_start (bytes_lo) at once and the others (bytes_hi) once the tile
    // rows have been read.  Without reserved rows, lo_start = 0.
    int buf_rows;
    int lo_start;
    unsigned bytes_lo, bytes_hi;
};

constexpr int kTileRows = 128;                    // a tile's own rows of one tensor (two 64-row boxes)

// reserve_rows: buffer rows [0, reserve_rows) hold the tile's own rows first
// (a multiple of kTileRows; see MmaLayout).
bool build_mma_layout(const Shape& s, const RungParams& r, double rope_base, size_t smem_limit, MmaLayout* L,
                      int reserve_rows = 0);
// Key-centric counterpart: query rows [0, M+1+Wp) and [s0, s0+M+1) relative to
// the first key of a tile (win_smem: relative row 0; rung_smem[k]: row s0_k).
bool build_key_layout(const Shape& s, const RungParams& r, double rope_base, size_t smem_limit, MmaLayout* L);
size_t fwd_mma_smem_bytes(const MmaLayout& L);
// Static shared memory of a forward CTA of one team (8 warps).
size_t fwd_mma_static_smem();
// Dynamic shared memory a grouped-query forward CTA may use (keys and values
// both resident).
size_t fwd_mma_gqa_smem_limit();
// 3-D tensor map [heads][T][64] of 2-byte rows, boxes of box_rows rows,
// 128-byte swizzle; rows outside [0, T) read as zero.
bool encode_rows_map(CUtensorMap* map, const void* base, CUtensorMapDataType dt, int T, int heads, int box_rows);

// A staged tensor: the same rows as 64-row and as 8-row boxes.
struct RowMaps { CUtensorMap m64, m8; };
inline bool encode_row_maps(RowMaps* m, const void* base, CUtensorMapDataType dt, int T, int heads) {
    return encode_rows_map(&m->m64, base, dt, T, heads, 64) && encode_rows_map(&m->m8, base, dt, T, heads, 8);
}
// The query backward's tile rows: q, dO, o (64-row loads) and the rotated q
// it writes back (40-row stores).
struct QTileMaps { CUtensorMap q, g, o, qt; };
cudaError_t launch_fwd_mma(const FwdArgs& a, const MmaLayout& L, cudaStream_t st);

// Tensor-core query-centric backward over the same staged rows (bf16 I/O;
// needs the forward output for Delta).  Its CTAs write rung partials as
// columns [0, bwd_mma_blocks) of BwdArgs::rpart; static shared memory is
// bwd_mma_static_smem() bytes on top of fwd_mma_smem_bytes(L).
size_t bwd_mma_static_smem();
int bwd_mma_blocks(const Shape& s);
cudaError_t launch_bwd_query_mma(const BwdArgs& a, const MmaLayout& L, cudaStream_t st);
// Tensor-core key-centric backward: dv and dk from the {p, dS} pairs of the
// tensor-core query pass, staging q~ and dO rows of the layout above.
int bwd_key_mma_blocks(const Shape& s);
// Dynamic shared memory of the key pass (the staged rows).
size_t bwd_key_mma_smem_bytes(const MmaLayout& L, bool saved);
size_t bwd_key_mma_static_smem();
cudaError_t launch_bwd_key_mma(const BwdArgs& a, const MmaLayout& L, cudaStream_t st);

}  // namespace fibattn
