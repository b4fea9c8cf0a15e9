// Launch shapes of the CPDP kernels: how many blocks a launch gets and, per
// reconcile variant, the rows per load chunk, the resident blocks per SM it is
// compiled for and when it loads the anchor and velocity. Kept apart from the C
// ABI's host code because, with the kernels in cpdp_kernels.cuh, these decide
// what each launch does on the GPU.
#pragma once

#include <cstdint>
#include <type_traits>

#include "cpdp_kernels.cuh"

namespace cpdp {

constexpr int kLocalUnroll = 2;  // float4 vectors per thread per iteration in the local step
constexpr int64_t kMaxGrid = 0x7fffffff;

// Blocks for `work_items` items at `per_block` items per block (kernels loop
// over any remainder beyond the grid limit).
inline unsigned grid_for(int64_t work_items, int64_t per_block) {
    int64_t blocks = (work_items + per_block - 1) / per_block;
    if (blocks < 1) blocks = 1;
    if (blocks > kMaxGrid) blocks = kMaxGrid;
    return static_cast<unsigned>(blocks);
}

// Rows per load chunk of the vectorised reconcile, the resident blocks per SM it
// is compiled for (3 blocks of 256 threads: 80 registers; 4 blocks: 64) and
// whether theta_ref and v are loaded after the rows (late) to free registers.
// Each entry is the fastest measured (ResNet-50 or ViT-S shape, W = 8, TB/s).
// SGD, float32 gradients: 4 rows, 3 blocks, early (7.00; late 6.95).
// SGD, bf16: 2 rows, 4 blocks, late (6.84; 3 rows / 3 blocks early 6.73).
// SGD with state reconciliation (two more running sums): 1 row, 4 blocks, late
// (7.00; early 6.97; 2 rows / 3 blocks 6.25).
// AdamW carries a third state row per worker. float32 gradients: 1 row,
// 4 blocks, early (6.71; late 6.67). bf16: 2 rows, 4 blocks, late (6.65, with a
// 20-byte spill; 1 row early 6.53). With state reconciliation: 2 rows, 4 blocks,
// late (after the AdamW step moved to the fast division; W = 8, ViT-S bf16 6.78
// against 6.56 at 1 row, ResNet-50 float32 6.77 against 6.54; W = 16 6.69 and
// 6.54 against 6.32 and 6.31).
template <int OPT, typename G, bool SS>
struct ReconcileShape {
    static constexpr int rows = 1, min_blocks = 4;
    static constexpr bool late = true;
};
template <>
struct ReconcileShape<kOptSGD, float, false> {
    static constexpr int rows = 4, min_blocks = 3;
    static constexpr bool late = false;
};
template <>
struct ReconcileShape<kOptSGD, bf16_bits, false> {
    static constexpr int rows = 2, min_blocks = 4;
    static constexpr bool late = true;
};
template <>
struct ReconcileShape<kOptAdamW, float, false> {
    static constexpr int rows = 1, min_blocks = 4;
    static constexpr bool late = false;
};
template <>
struct ReconcileShape<kOptAdamW, bf16_bits, false> {
    static constexpr int rows = 2, min_blocks = 4;
    static constexpr bool late = true;
};
template <typename G>
struct ReconcileShape<kOptAdamW, G, true> {
    static constexpr int rows = 2, min_blocks = 4;
    static constexpr bool late = true;
};

// Two workers: 2-row chunks fill every slot, and the freed registers allow 4
// resident blocks. Measured at N = 2^26 (TB/s, against the shapes above):
// SGD float32 7.03 (6.67), AdamW float32 6.79 late (6.43), SGD with state
// reconciliation 7.00 early (6.34), AdamW with state reconciliation 5.96 late
// (5.64); the bf16 SGD and AdamW shapes above already use 2 rows.
template <int OPT, typename G, bool SS>
struct ReconcileShapeW2 {
    static constexpr int rows = 2, min_blocks = 4;
    static constexpr bool late = OPT == kOptAdamW || (!SS && !std::is_same<G, float>::value);
};

// Three to six workers: the general shapes, except SGD with bf16 gradients,
// where 3-row chunks at 3 blocks with early anchor loads measured fastest
// (N = 2^25, TB/s against 2 rows: W = 3 6.75 / 6.14, W = 4 6.63 / 6.55,
// W = 5 6.88 / 6.38, W = 6 6.95 / 6.64; from W = 7 on the 2-row shape is as
// fast or faster).
template <int OPT, typename G, bool SS>
struct ReconcileShapeFew : ReconcileShape<OPT, G, SS> {};
template <>
struct ReconcileShapeFew<kOptSGD, bf16_bits, false> {
    static constexpr int rows = 3, min_blocks = 3;
    static constexpr bool late = false;
};

// One worker (no state reconciliation, which has nothing to average): 1-row
// chunks at 4 resident blocks with early anchor loads measured fastest at
// N = 2^26 (TB/s, against the general shapes): SGD float32 6.51 (5.73), SGD
// bf16 6.29 (5.71), AdamW bf16 6.29 (5.59); AdamW float32 already uses it.
struct ReconcileShapeW1 {
    static constexpr int rows = 1, min_blocks = 4;
    static constexpr bool late = false;
};

}  // namespace cpdp
