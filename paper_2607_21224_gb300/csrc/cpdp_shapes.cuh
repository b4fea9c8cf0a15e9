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

// The local step's vectors per thread run along the warp (each warp streams
// 1 KB of every array) for AdamW with bf16 gradients: 7,157 against 7,035 GB/s
// (ViT-S N, W = 8, back-to-back launches; 7,118 against 7,002 at the ResNet-50
// N). The other variants measured the same or up to 1 % slower that way and
// keep a block-wide spacing.
template <int OPT, typename G>
struct LocalWarpRuns {
    static constexpr bool value = OPT == kOptAdamW && !std::is_same<G, float>::value;
};
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
// is compiled for (3 blocks of 256 threads: 80 registers; 4 blocks: 64),
// whether theta_ref and v are loaded after the rows (late) to free registers,
// and whether its offsets are 32-bit where the sizes allow (narrow), which
// frees more. Each entry is the fastest measured (ResNet-50 or ViT-S shape,
// W = 8, TB/s).
// SGD, float32 gradients: 4 rows, 3 blocks, early (7.00; late 6.95; narrow
// offsets make no difference).
// SGD, bf16: 2 rows, 4 blocks, late (6.84; 3 rows / 3 blocks early 6.73; narrow
// 0.8 % slower).
// SGD with state reconciliation (two more running sums): 1 row, 4 blocks, late
// (7.00; early 6.97; 2 rows / 3 blocks 6.25; narrow 1 % slower).
// AdamW carries a third state row per worker. With 64-bit offsets its 2-row
// shape at 4 blocks spilled 24-32 bytes; narrow offsets remove the spill:
// 2 rows, 4 blocks, late, narrow for every AdamW variant (CPDP and DDP without
// state reconciliation now take the gradient-chunk shapes below). Isolated launches at
// the ViT-S N (GB/s, against the best 64-bit shape): bf16 gradients 6,818
// (6,605), float32 6,785 (6,730 at 1 row, early), with state reconciliation
// 6,541 (6,467, bf16) and 6,427 (6,337, float32); at W = 16 +2 to +3 %.
template <int OPT, typename G, bool SS>
struct ReconcileShape {
    static constexpr int rows = 2, min_blocks = 4;
    static constexpr bool late = true, narrow = true;
};
template <>
struct ReconcileShape<kOptSGD, float, false> {
    static constexpr int rows = 4, min_blocks = 3;
    static constexpr bool late = false, narrow = false;
};
template <>
struct ReconcileShape<kOptSGD, bf16_bits, false> {
    static constexpr int rows = 2, min_blocks = 4;
    static constexpr bool late = true, narrow = false;
};
template <typename G>
struct ReconcileShape<kOptSGD, G, true> {
    static constexpr int rows = 1, min_blocks = 4;
    static constexpr bool late = true, narrow = false;
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
    static constexpr bool narrow = OPT == kOptAdamW;
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
    static constexpr bool late = false, narrow = false;
};

// Three-row chunks at 4 resident blocks (late anchor, narrow offsets) for
// worker counts they divide or nearly divide, where they measured at least 2 %
// faster than the shapes above (20 back-to-back launches at N = 2^25, GB/s
// against the shape used before). W = 3: CPDP SGD bf16 6,593 (6,376), CPDP
// SGD with state reconciliation f32 6,562 (5,923) and bf16 6,187 (5,594), DDP
// SGD f32 7,113 (6,680); CPDP AdamW bf16 also measured faster there (6,211
// against 6,096) and now takes the gradient-chunk shape below. W = 5: DDP SGD
// f32 7,081 (6,765). W = 6: CPDP SGD with state reconciliation f32 6,989 (6,867)
// and bf16 6,768 (6,610), DDP SGD f32 7,090 (6,949). Through the library
// (N = 2^25, K = 2, sync-step GB/s) the W = 3 entries gained 1.5-12 % and the
// W = 5 DDP entry 2.6 %; DDP AdamW bf16 at W = 3, which the launch-by-launch
// probe also favoured, lost 2.9 % there and keeps the one-pass kernel.
template <int METHOD, int OPT, bool SS, typename G, int W>
struct ReconcileThreeRows {
    static constexpr bool use = false;
    static constexpr int rows = 3, min_blocks = 4;
    static constexpr bool late = true, narrow = true;
};
#define CPDP_THREE_ROWS(M, O, SS, G, W)                      \
    template <>                                              \
    struct ReconcileThreeRows<M, O, SS, G, W> {              \
        static constexpr bool use = true;                    \
        static constexpr int rows = 3, min_blocks = 4;       \
        static constexpr bool late = true, narrow = true;    \
    };
CPDP_THREE_ROWS(kMethodCPDP, kOptSGD, false, bf16_bits, 3)
CPDP_THREE_ROWS(kMethodCPDP, kOptSGD, true, float, 3)
CPDP_THREE_ROWS(kMethodCPDP, kOptSGD, true, bf16_bits, 3)
CPDP_THREE_ROWS(kMethodDDP, kOptSGD, false, float, 3)
CPDP_THREE_ROWS(kMethodDDP, kOptSGD, false, float, 5)
CPDP_THREE_ROWS(kMethodCPDP, kOptSGD, true, float, 6)
CPDP_THREE_ROWS(kMethodCPDP, kOptSGD, true, bf16_bits, 6)
CPDP_THREE_ROWS(kMethodDDP, kOptSGD, false, float, 6)
#undef CPDP_THREE_ROWS

// Gradient-row chunks, for AdamW and for SGD with bf16 gradients (CPDP and
// DDP without state reconciliation; CPDP AdamW with state reconciliation at 3
// to 5 workers): the gradient rows in chunks of 8 (bf16) or 4 (float32) held
// as raw words, the first state chunk loaded together with the first gradient
// chunk, then the state rows in chunks (narrow offsets, late anchor). The
// results are bit-identical to those of the other shapes. Isolated launches
// at the ViT-S N (W = 32 at N / 2), GB/s against the shape used before:
// AdamW from 2 workers (CPDP; float32 gradients at W = 2 keep the one-pass
// kernel, within 0.4 %; DDP from 5, where the one-pass kernel does not take
// W = 2-4), 2-row state chunks at 4 blocks up to 7 workers and 3-row chunks at
// 3 blocks from 8. CPDP bf16 gradients W = 2 (N = 2^26) 6,987 (6,772; one-pass
// 6,765), W = 3 6,922 (6,600, three-row shape), W = 4 7,008 (6,782), W = 5
// 6,963 (6,600), W = 6 6,965 (6,809),
// W = 7 6,967 (6,904), W = 8 6,979 (6,931; 2-row 6,966), W = 12 6,941 (6,859;
// 2-row 6,911), W = 16 6,917 (6,852), W = 32 6,838 (6,791); float32 gradients
// W = 3 6,997 (6,569), W = 4 7,067 (6,934), W = 5 6,979 (6,755), W = 6 6,998
// (6,928), W = 7 7,004 (6,882), W = 8 7,021 (6,926; 2-row 7,011), W = 12 6,995
// (6,888), W = 16 6,948 (6,853), W = 32 6,899 (6,833); DDP +1 to +6 % at
// W = 5-16. DDP at W = 3-4 measured within 1.3 % of its one-pass kernel.
// AdamW with state reconciliation (CPDP), 2-row chunks at 4 blocks for 3 to 5
// workers: bf16 gradients W = 3 6,496 (6,155), W = 4 6,758 (6,561), W = 5
// 6,665 (6,380); float32 W = 3 6,729 (6,344), W = 4 6,871 (6,777), W = 5 6,703
// (6,570); from W = 6 the shapes above measured as fast or faster.
// SGD with bf16 gradients, 4-row state chunks at 3 blocks, CPDP from 7
// workers (W = 7 7,007 (6,773), W = 8 7,031 (6,913), W = 12 6,976 (6,783),
// W = 16 6,969 (6,886), W = 32 6,891 (6,847); at W = 5-6 within 0.3 %), DDP
// from 5 (W = 5 +5.8 %, W = 6 +1.6 %, W = 8 +4.5 %, W = 16 +5.4 %). With
// float32 gradients the SGD shapes gain at most 0.2 % (CPDP) and 0.6 % (DDP),
// and with state reconciliation nothing, so those keep their shapes.
// The same row traffic in a plain local step walked column by column (no
// sums, no dependency between the rows) peaks at 6,999 GB/s at W = 8 (4-row
// chunks, 2 blocks; 6,930 at 2 rows and 4 blocks), against 7,155 for the flat
// local step: the W = 8 AdamW shape is within 0.3 % of that floor.
// MANY selects the shape from kGradChunksManyWorkers workers on; the other
// one covers min_workers to max_workers (below kGradChunksManyWorkers).
constexpr int kGradChunksManyWorkers = 8;
template <int METHOD, int OPT, bool SS, typename G, bool MANY>
struct ReconcileGradChunks {
    static constexpr bool use = false;
};
template <int METHOD, typename G, bool MANY>
struct ReconcileGradChunks<METHOD, kOptAdamW, false, G, MANY> {
    static constexpr bool use = METHOD != kMethodLocalSGD;
    static constexpr int min_workers = METHOD == kMethodDDP ? 5 : 2, max_workers = kGradChunksManyWorkers - 1;
    static constexpr int rows = MANY ? 3 : 2, min_blocks = MANY ? 3 : 4;
    static constexpr int grad_rows = std::is_same<G, float>::value ? 4 : 8;
    static constexpr bool late = true, narrow = true, overlap = true;
};
template <typename G, bool MANY>
struct ReconcileGradChunks<kMethodCPDP, kOptAdamW, true, G, MANY> {
    static constexpr bool use = !MANY;
    static constexpr int min_workers = 3, max_workers = 5;
    static constexpr int rows = 2, min_blocks = 4, grad_rows = std::is_same<G, float>::value ? 4 : 8;
    static constexpr bool late = true, narrow = true, overlap = true;
};
template <int METHOD, bool MANY>
struct ReconcileGradChunks<METHOD, kOptSGD, false, bf16_bits, MANY> {
    static constexpr bool use = METHOD != kMethodLocalSGD;
    static constexpr int min_workers = METHOD == kMethodDDP ? 5 : 7, max_workers = kGradChunksManyWorkers - 1;
    static constexpr int rows = 4, min_blocks = 3, grad_rows = 8;
    static constexpr bool late = true, narrow = true, overlap = true;
};

// Gradient rows per chunk and overlap of a shape: its own where it states
// them, else the state-row chunk and no overlap.
template <typename S, typename = void>
struct GradChunkOf {
    static constexpr int rows = S::rows;
    static constexpr bool overlap = false;
};
template <typename S>
struct GradChunkOf<S, std::void_t<decltype(S::grad_rows)>> {
    static constexpr int rows = S::grad_rows;
    static constexpr bool overlap = S::overlap;
};

// One round trip for few workers (reconcile_onepass_kernel: every row of a
// column loaded before any is used). Where it is used, and at how many
// resident blocks, per method, optimizer, state reconciliation and gradient
// type: each entry measured at least 2 % faster than the shapes above at
// N = 2^26 (GB/s, against the vec4 kernel). Entries not listed keep the vec4
// kernel.
// One worker, every variant: 1 row, 4 blocks. CPDP SGD f32 6,788 (5,620),
// SGD bf16 6,483 (5,385), AdamW f32 6,866 (5,814), AdamW bf16 6,653 (5,642);
// LocalSGD and DDP 6,004-6,848 (4,411-6,005); state reconciliation 3,967-5,603
// (3,519-4,189).
struct OnePassW1 {
    static constexpr bool use = true;
    static constexpr int wmax = 1, min_blocks = 4;
};
template <int METHOD, int OPT, bool SS, typename G>
struct OnePassW2 {
    static constexpr bool use = false;
    static constexpr int wmax = 2, min_blocks = 4;
};
// Two workers. CPDP: SGD f32 7,064 (6,792), SGD bf16 6,979 (5,958), AdamW f32
// 7,023 (6,422); with state reconciliation SGD f32 6,344 (6,116), SGD bf16
// 6,768 (5,197), AdamW f32 6,018 (5,364), AdamW bf16 at 3 blocks 5,411
// (5,073). DDP: SGD f32 7,059 (6,694), SGD bf16 6,945 (6,023), AdamW f32 at 3
// blocks 6,901 (6,748), AdamW bf16 6,960 (6,152). CPDP AdamW bf16 without state
// reconciliation and LocalSGD measured as fast or faster with the vec4 kernel.
#define CPDP_ONEPASS(NAME, M, O, SS, G, BLOCKS)          \
    template <>                                         \
    struct NAME<M, O, SS, G> {                          \
        static constexpr bool use = true;               \
        static constexpr int wmax = NAME##Max, min_blocks = BLOCKS; \
    };
constexpr int OnePassW2Max = 2;
CPDP_ONEPASS(OnePassW2, kMethodCPDP, kOptSGD, false, float, 4)
CPDP_ONEPASS(OnePassW2, kMethodCPDP, kOptSGD, false, bf16_bits, 4)
CPDP_ONEPASS(OnePassW2, kMethodCPDP, kOptAdamW, false, float, 4)
CPDP_ONEPASS(OnePassW2, kMethodCPDP, kOptSGD, true, float, 4)
CPDP_ONEPASS(OnePassW2, kMethodCPDP, kOptSGD, true, bf16_bits, 4)
CPDP_ONEPASS(OnePassW2, kMethodCPDP, kOptAdamW, true, float, 4)
CPDP_ONEPASS(OnePassW2, kMethodCPDP, kOptAdamW, true, bf16_bits, 3)
CPDP_ONEPASS(OnePassW2, kMethodDDP, kOptSGD, false, float, 4)
CPDP_ONEPASS(OnePassW2, kMethodDDP, kOptSGD, false, bf16_bits, 4)
CPDP_ONEPASS(OnePassW2, kMethodDDP, kOptAdamW, false, float, 3)
CPDP_ONEPASS(OnePassW2, kMethodDDP, kOptAdamW, false, bf16_bits, 4)

// Three workers (4-row chunk, the kernel skips the fourth). CPDP SGD f32
// 7,075 (6,731); LocalSGD SGD bf16 6,972 (6,666); DDP SGD bf16 6,985 (6,255),
// AdamW f32 7,018 (6,358), AdamW bf16 at 2 blocks 6,207 (5,974).
template <int METHOD, int OPT, bool SS, typename G>
struct OnePassW3 {
    static constexpr bool use = false;
    static constexpr int wmax = 4, min_blocks = 3;
};
constexpr int OnePassW3Max = 4;
CPDP_ONEPASS(OnePassW3, kMethodCPDP, kOptSGD, false, float, 3)
CPDP_ONEPASS(OnePassW3, kMethodLocalSGD, kOptSGD, false, bf16_bits, 3)
CPDP_ONEPASS(OnePassW3, kMethodDDP, kOptSGD, false, bf16_bits, 3)
CPDP_ONEPASS(OnePassW3, kMethodDDP, kOptAdamW, false, float, 3)
CPDP_ONEPASS(OnePassW3, kMethodDDP, kOptAdamW, false, bf16_bits, 2)

// Four workers. CPDP SGD bf16 at 2 blocks 6,803 (6,258); LocalSGD SGD bf16
// 7,005 (6,705); DDP SGD bf16 7,004 (6,174), AdamW f32 6,992 (6,749), AdamW
// bf16 at 2 blocks 6,758 (6,419).
template <int METHOD, int OPT, bool SS, typename G>
struct OnePassW4 {
    static constexpr bool use = false;
    static constexpr int wmax = 4, min_blocks = 3;
};
constexpr int OnePassW4Max = 4;
CPDP_ONEPASS(OnePassW4, kMethodCPDP, kOptSGD, false, bf16_bits, 2)
CPDP_ONEPASS(OnePassW4, kMethodLocalSGD, kOptSGD, false, bf16_bits, 3)
CPDP_ONEPASS(OnePassW4, kMethodDDP, kOptSGD, false, bf16_bits, 3)
CPDP_ONEPASS(OnePassW4, kMethodDDP, kOptAdamW, false, float, 3)
CPDP_ONEPASS(OnePassW4, kMethodDDP, kOptAdamW, false, bf16_bits, 2)
#undef CPDP_ONEPASS

}  // namespace cpdp
