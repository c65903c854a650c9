// cci_gemm_ws.cuh -- the dense tensor-core product of the workspace family
// (CCI_ALGO_DENSE_TC_WS) after the one-pass decompression of the packed weights.
//
// D[n][co] = sum_r x[n][r] * Wd[co][r] on tcgen05 with fp32 accumulators in TMEM,
// tile [128 n][BN co], BN in {64, 128, 256}, two BN-column accumulators:
//   bf16:  A = activation tile [128 n][64 r], B = weight tile [BN co][64 r], one
//          kind::f16 MMA per 16 r.
//   fp32 layers: every operand split as hi + lo (hi a tf32 value, lo = v - hi
//          exactly; cci_common.cuh), 32 r per stage and 8 MMAs: hi(x) hi(w) as
//          four kind::tf32 MMAs, bf16(x) bf16(lo(w)) and bf16(lo(x)) bf16(hi(w))
//          as two kind::f16 MMAs each; operand plane 0 holds hi, plane 1 the
//          bf16 pairs (a 128-byte row per stage: 32 bf16 of one term, then 32 of
//          the other).
// Operands (all K-major, 128-byte swizzle, 1024-byte aligned stage buffers):
//   weights      TMA from the workspace planes (tensor maps over [Cout][R], fp32
//                plane 1 over [Cout][ceil(R / 32) * 64] bf16);
//   activations  one of (the template's ASRC):
//     kA2d      products: TMA over X[N][Cin];
//     kA4d      stride-1 convolutions with Cin a multiple of the stage depth:
//               TMA over X[B][H][W][Cin] with a box of QB x PB x BB output
//               pixels (QB*PB*BB <= 128 rows), shifted by the tap (kh, kw); the
//               zero padding is the copy's out-of-range fill;
//     kAHalo    bf16 3x3 convolutions with unit stride and padding 1: per tile
//               and 64-channel chunk one TMA copy of the input halo, rows
//               (p, q) of PB input rows + 2 by Q + 2 columns (the padding is the
//               copy's out-of-range fill); the tile's output rows are laid out on
//               the same Q + 2 wide grid (two unused columns per row), so tap
//               (kh, kw) reads the halo from row kh * (Q + 2) + kw on: the A
//               operand of every tap is the same buffer at a row offset (the
//               128-byte swizzle follows the address, so any row offset works);
//               per stage only the tap's weight tile is copied (CTA pairs: each
//               CTA copies its own halo and half of the weight rows, both CTAs'
//               copies completing on the even CTA's barriers);
//     kAGather  other convolutions: the producer warps gather rows (cp.async for
//               bf16; registers, two stages ahead, then the hi/lo split, for fp32).
//   fp32 activations copied by TMA land raw in shared memory; the producer warps
//   split each row and store its two planes in tensor memory (per stage 64
//   columns after the accumulators: 32 of tf32 hi, 16 of bf16 pairs of x, 16 of
//   lo(x)), from where the MMAs read A: the eight MMAs then read only B from
//   shared memory.
// Weights (the template's PK):
//   PK = false  the dense workspace planes written by the one-pass decompression;
//   PK = true   the packed (value, index) pairs themselves (bf16 only, no
//               workspace): two groups of four producer warps take the stages
//               in turn; each thread loads the K-slot runs of its groups from
//               global memory two of its stages ahead (into registers), expands
//               them into rows (Alg. 2's index: each pair goes to row G*i + Idx
//               of its group), 8 rows x 8 indices per thread, and once the stage
//               is free stores the rows into its swizzled B tile.
// Output: Y (fp32, or bf16 with the fused epilogue's bias and ReLU) written by
// TMA stores from swizzled staging buffers of [128 rows][128 bytes] (two per
// epilogue group, four in the two-group form with N tiles up to 128), 2-D over
// Y[N][Cout] or, for kA4d and kAHalo, 4-D over Y[B][P][Q][Cout] with the tile's
// pixel box.
// Roles: warps 0-3 epilogue (TMEM lanes), warps 4-7 producers of the activation
// planes that are not copied by TMA (PK: of the weight tiles, with warps
// 9 + kIssuers .. + 3 as the second producer group), warp 8 allocates TMEM and
// issues the MMAs, warps 9 .. 8 + kIssuers issue the TMA copies as soon as a
// stage is free (so copy latency overlaps the producers' work), stage by stage in
// turn: the copies one thread issues are processed one box after another
// (measured on GB300: about 0.5 us per box of 16-64 KB from one issuer; copy
// throughput grows with the number of issuing warps), so up to six warps issue
// (one per stage in flight; PK: three, one activation box per stage).  Every
// mbarrier wait is bounded (CCI_ERR_TIMEOUT, abort flag, drain, TMEM freed).
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>

#include <type_traits>

#include "cci_tc_common.cuh"

namespace cci {
namespace ws {

enum ASrc { kA2d = 0, kA4d = 1, kAGather = 2, kAHalo = 3 };

// output-pixel box of one M tile of a convolution whose activations are copied
// by 4-D TMA: rows m = (bi*PB + pi)*QB + qi of the tile are the pixels
// (b0 + bi, p0 + pi, q0 + qi); rows >= QB*PB*BB are unused.  Halo copies: QB = Q,
// BB = 1, rows m = pi*(Q + 2) + qi (qi >= Q unused), rows = PB*(Q + 2)
struct ConvBox {
    int QB, PB, BB;  // box extent along q, p and the batch
    int nQ, nP;      // boxes along q and p (the batch index is the rest)
    int rows;        // QB * PB * BB
    int64_t B;       // batch size
    int hrows;       // halo copies: rows of one halo buffer (a multiple of 8)
    int nh;          // halo copies: buffers in the ring (0 otherwise)
    int resident;    // halo copies: the layer's whole weight matrix stays in the stages
                     // (one N tile, every stage of a tile a stage of the ring): the
                     // weights are copied for the CTA's first tile only
};

// activation tensor maps: [0] for products (2-D over X[N][Cin]); for a
// convolution with strides (sh, sw) <= 2, map [rh * sw + rw] covers the input
// pixels (h, w) = (rh + sh * h', rw + sw * w'), a 4-D tensor over (ci, w', h', b)
struct AMaps {
    CUtensorMap m[4];
};

// CG = 2: a cluster of two CTAs computes a 256 x BN tile with tcgen05.mma
// cta_group::2 issued by the even CTA; each CTA holds its 128 rows of A and half
// of the BN rows of B (bf16 with TMA activations only)
// EPI = 2: a second epilogue group (warps 4-7, idle when bf16 activations are
// copied by TMA) and two staging buffers per group, for layers whose tiles have
// few stages (the output write dominates); EPI = 1: one group, more stages
template <bool TF32, int ASRC, int BN, int CG, int EPI, bool PK = false, bool MC = false>
struct Cfg {
    static constexpr int kM = 128, kN = BN;
    static_assert(CG == 1 || (CG == 2 && !TF32 && ASRC != kAGather), "pair mode: bf16 with TMA activations");
    static_assert(!PK || (!TF32 && ASRC != kAGather && EPI == 1 && (BN / CG) <= 128),
                  "packed weights: bf16, TMA activations, producers busy, one item per producer");
    static constexpr int kBRows = kN / CG;  // B rows held by one CTA
    // MC: a cluster of two CTAs takes adjacent M tiles of the same N tile; each
    // copies half of the B rows of a stage with multicast into both, and each
    // CTA's MMAs release the stage in both (TMA activations, 2-D or 4-D)
    static_assert(!MC || (ASRC != kAGather && ASRC != kAHalo && CG == 1 && EPI == 1 && !PK),
                  "weight multicast: single-CTA TMA tiles with one epilogue group");
    // (used for fp32 layers: measured on the bf16 3x3 convolutions it did not pay,
    // conv3x3_28 0.0273 -> 0.0283 ms, the ResNet-50 stack unchanged)
    static constexpr bool kPairUnits = CG == 2 || MC;  // units of two M tiles over a cluster of two
    static constexpr int kKS = TF32 ? 32 : 64;  // r per stage: one 128-byte row
    static constexpr bool kATma = !TF32 && ASRC != kAGather;  // A copied by TMA into its plane
    static constexpr bool kHalo = ASRC == kAHalo;  // A: per-chunk halo buffers, stages hold B only
    static_assert(!kHalo || (!TF32 && (CG == 1 || !PK)), "halo copies: bf16 tiles (pairs: workspace weights)");
    // raw fp32 A by TMA; the producers split it into its two planes and write both to
    // tensor memory, where the MMAs read A (no A planes in shared memory)
    static constexpr bool kARaw = TF32 && ASRC != kAGather;
    static constexpr int kAPlanes = (TF32 && !kARaw) ? 2 : 1, kBPlanes = TF32 ? 2 : 1;
    static constexpr int kAPlane = kM * 128;                    // bytes: 128-byte rows
    static constexpr int kBPlane = kBRows * 128;
    static constexpr int kBOff = kHalo ? 0 : kAPlanes * kAPlane;  // B planes within a stage
    static constexpr int kStage = kBOff + kBPlanes * kBPlane;
    static_assert(kStage % 1024 == 0, "stages must keep the 1024-byte swizzle alignment");
    // halo copies: fewer weight stages, the rest of shared memory for a ring of
    // halo buffers whose size and count the host sets per layer (ConvBox)
    // (9 stages of 8 KB: a 3x3 layer of 64 input and 64 output channels keeps its
    // weights resident)
    static constexpr int kHaloStages = kBPlane <= 8192 ? 9 : (kBPlane <= 16384 ? 4 : 3);
    static constexpr int kYBuf = kM * 128;  // one output staging buffer: [128 rows][32 fp32]
    // epilogue groups: warps 0-3, and warps 4-7 too when they have no producer work
    // (TMA-copied bf16 activations); two staging buffers per group, four in the
    // two-group form with N tiles up to 128 (short tiles, bound by the output
    // write: more stores in flight, three or four stages are enough)
    static constexpr int kEG = (kATma && EPI == 2) ? 2 : 1;
    static constexpr int kYPerGroup = (kEG == 2 && BN <= 128) ? 4 : 2;
    static constexpr int kYBufs = kYPerGroup * kEG;
    static_assert(EPI == 1 || EPI == 2, "epilogue groups");
    static constexpr int kBudget = static_cast<int>(kMaxSmemPerBlock) - 1024 - kYBufs * kYBuf - 1024;
    static constexpr int kStagesFit = (kBudget / kStage) < tc::kMaxStages ? (kBudget / kStage) : tc::kMaxStages;
    static constexpr int kStages = kHalo ? kHaloStages : kStagesFit;
    // accumulators: 2 x kN columns; kARaw adds per stage the A planes (32 + 32 columns)
    static constexpr int kAColBase = 2 * kN;
    static constexpr int kTmemCols = kARaw ? 512 : 2 * kN;
    static constexpr size_t kSmem =
        1024 + static_cast<size_t>(kStages) * kStage + kYBufs * kYBuf + sizeof(tc::Smem) + 64;  // + halo ring
    static constexpr uint32_t kBBytes = kBPlanes * kBPlane;
    static constexpr uint32_t kIdesc = (1u << 4)                                           // D f32
                                       | (TF32 ? (2u << 7) | (2u << 10) : (1u << 7) | (1u << 10))  // tf32 / bf16
                                       | (static_cast<uint32_t>(kN >> 3) << 17) |
                                       (static_cast<uint32_t>((kM * CG) >> 4) << 24);
    // fp32 layers: the bf16 MMAs of the split's cross terms
    static constexpr uint32_t kIdescB = (1u << 4) | (1u << 7) | (1u << 10) | (static_cast<uint32_t>(kN >> 3) << 17) |
                                        (static_cast<uint32_t>((kM * CG) >> 4) << 24);
    static_assert(kSmem <= kMaxSmemPerBlock, "stage buffers over the per-block limit");
    static_assert(kStages >= 3, "too few pipeline stages");
    static_assert(kTmemCols == 128 || kTmemCols == 256 || kTmemCols == 512, "TMEM allocation not a power of 2");
    static_assert(!kARaw || kAColBase + kStages * 64 <= 512, "A stages do not fit in tensor memory");
    // warps issuing the TMA copies, stage `it` by warp 9 + it % kIssuers: one
    // thread's copies are processed one box at a time, so several issuers keep
    // more boxes moving.  kIssuers <= kStages keeps every empty-barrier wait
    // within one phase of the barrier (no parity aliasing).
    // (kAHalo: one more warp, which copies the halos)
    // PK: three issuers (one activation box per stage) and a second group of four
    // producer warps after them
    static constexpr int kStageIssuers = PK ? (kHalo ? 1 : 3) : 6;  // PK halo stages: the producers' tiles only
    static constexpr int kIssuers =
        ASRC == kAGather ? 1 : (kStages < kStageIssuers ? kStages : kStageIssuers) + (kHalo ? 1 : 0);
    static constexpr int kProdGroups = PK ? 2 : 1;
    static constexpr int kThreads = 32 * (9 + kIssuers + 4 * (kProdGroups - 1));
    static_assert(kIssuers - (kHalo ? 1 : 0) >= 1 && kIssuers - (kHalo ? 1 : 0) <= kStages,
                  "stage issuers must not outnumber the stages");
};

template <bool TF32, int CG>
__device__ __forceinline__ void mma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc)
{
    if constexpr (CG == 2) {
        asm volatile(
            "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
            "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
            "l"(a), "l"(b), "r"(idesc), "r"(acc)
            : "memory");
    } else if constexpr (TF32) {
        asm volatile(
            "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
            "tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
            "l"(a), "l"(b), "r"(idesc), "r"(acc)
            : "memory");
    } else {
        asm volatile(
            "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
            "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
            "l"(a), "l"(b), "r"(idesc), "r"(acc)
            : "memory");
    }
}

// ---- one pipeline stage of the fp32 product (8 MMAs), A in tensor memory ----
// The three terms of the split (cci_common.cuh) over a 32-wide stage:
//   hi(x) hi(w)           4 kind::tf32 MMAs: A at TMEM columns a0 + 8k, B plane 0
//                         at descriptor b0 + 2k (32 bytes per 8 indices);
//   bf16(x) bf16(lo(w))   2 kind::f16 MMAs: A at a0 + 32 + 8k (two bf16 per
//                         column), B plane 1 (kB1 16-byte units on) at + 4 + 2k;
//   bf16(lo(x)) bf16(hi(w)) 2 kind::f16 MMAs: A at a0 + 48 + 8k, B plane 1 at + 2k.
// Every lane of the MMA warp executes the block; the lane with `issue` set issues
// the eight MMAs and commits the stage to `bar`.  One block with the addresses
// formed by adds: the MMA warp's instruction stream per stage bounds this
// product (measured on GB300 with clock stamps for the three-pass form of twelve
// MMAs: operands waited for ~130 cycles per stage, the issue of a stage took ~850).
// kMC: the commit arrives on the barrier at this offset in both CTAs of the cluster.
template <uint32_t kIdescT, uint32_t kIdescB, uint32_t kB1, bool kMC = false>
__device__ __forceinline__ void stage_tf32_split(uint32_t d, uint32_t a0, uint64_t b0, uint32_t acc0, uint32_t issue,
                                                 uint32_t bar)
{
    asm volatile(
        "{\n.reg .pred pe, pa, pt;\n.reg .b32 a;\n.reg .b64 b;\n"
        "setp.ne.b32 pe, %4, 0;\nsetp.ne.b32 pa, %3, 0;\nsetp.eq.b32 pt, 0, 0;\n"
        "@pe tcgen05.mma.cta_group::1.kind::tf32 [%0], [%1], %2, %5, pa;\n"
        "add.u32 a, %1, 8;\nadd.s64 b, %2, 2;\n"
        "@pe tcgen05.mma.cta_group::1.kind::tf32 [%0], [a], b, %5, pt;\n"
        "add.u32 a, %1, 16;\nadd.s64 b, %2, 4;\n"
        "@pe tcgen05.mma.cta_group::1.kind::tf32 [%0], [a], b, %5, pt;\n"
        "add.u32 a, %1, 24;\nadd.s64 b, %2, 6;\n"
        "@pe tcgen05.mma.cta_group::1.kind::tf32 [%0], [a], b, %5, pt;\n"
        "add.u32 a, %1, 32;\nadd.s64 b, %2, %7;\n"
        "@pe tcgen05.mma.cta_group::1.kind::f16 [%0], [a], b, %6, pt;\n"
        "add.u32 a, %1, 40;\nadd.s64 b, b, 2;\n"
        "@pe tcgen05.mma.cta_group::1.kind::f16 [%0], [a], b, %6, pt;\n"
        "add.u32 a, %1, 48;\nadd.s64 b, %2, %8;\n"
        "@pe tcgen05.mma.cta_group::1.kind::f16 [%0], [a], b, %6, pt;\n"
        "add.u32 a, %1, 56;\nadd.s64 b, b, 2;\n"
        "@pe tcgen05.mma.cta_group::1.kind::f16 [%0], [a], b, %6, pt;\n}\n" ::"r"(d),
        "r"(a0), "l"(b0), "r"(acc0), "r"(issue), "n"(kIdescT), "n"(kIdescB),
        "n"(static_cast<uint64_t>(kB1 + 4)), "n"(static_cast<uint64_t>(kB1))
        : "memory");
    if constexpr (kMC)
        asm volatile(
            "{\n.reg .pred pe;\nsetp.ne.b32 pe, %1, 0;\n"
            "@pe tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %2;\n}\n" ::"r"(bar),
            "r"(issue), "h"(static_cast<uint16_t>(3))
            : "memory");
    else
        asm volatile(
            "{\n.reg .pred pe;\nsetp.ne.b32 pe, %1, 0;\n"
            "@pe tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n}\n" ::"r"(bar),
            "r"(issue)
            : "memory");
}

// ---- one pipeline stage of bf16 MMAs ----
// Every lane of the MMA warp executes the block; the lane with `issue` set
// issues the four 16-deep MMAs of a 64-wide stage (descriptors advance by 32
// bytes, 2 units of 16 bytes, per MMA) and commits the stage to `bar`.  Kept in
// one block with the descriptors precomputed: the MMA warp's own instruction
// latency per stage bounds layers whose MMAs are short (measured on GB300: a
// 64-wide N tile stage is 192 tensor cycles, and the issue path was 400-700).
// kCounted: only the first n16 (1-4) MMAs of the stage, 16 reduction indices each
// (a one-stage layer copying fewer than 64 indices); else all four
template <uint32_t kIdesc, bool kMC = false, bool kCounted = false>
__device__ __forceinline__ void stage_f16(uint32_t d, uint64_t adesc, uint64_t bdesc, uint32_t acc0, uint32_t issue,
                                          uint32_t bar, uint32_t n16 = 4)
{
    if constexpr (kCounted)
        asm volatile(
            "{\n.reg .pred pe, pa, p1, p2, p3, pt;\n.reg .b64 ad, bd;\n"
            "setp.ne.b32 pe, %4, 0;\nsetp.ne.b32 pa, %3, 0;\nsetp.eq.b32 pt, 0, 0;\n"
            "setp.gt.and.u32 p1, %6, 1, pe;\nsetp.gt.and.u32 p2, %6, 2, pe;\nsetp.gt.and.u32 p3, %6, 3, pe;\n"
            "@pe tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %5, pa;\n"
            "add.s64 ad, %1, 2;\nadd.s64 bd, %2, 2;\n"
            "@p1 tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %5, pt;\n"
            "add.s64 ad, %1, 4;\nadd.s64 bd, %2, 4;\n"
            "@p2 tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %5, pt;\n"
            "add.s64 ad, %1, 6;\nadd.s64 bd, %2, 6;\n"
            "@p3 tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %5, pt;\n}\n" ::"r"(d),
            "l"(adesc), "l"(bdesc), "r"(acc0), "r"(issue), "n"(kIdesc), "r"(n16)
            : "memory");
    else
        asm volatile(
            "{\n.reg .pred pe, pa, pt;\n.reg .b64 ad, bd;\n"
            "setp.ne.b32 pe, %4, 0;\nsetp.ne.b32 pa, %3, 0;\nsetp.eq.b32 pt, 0, 0;\n"
            "@pe tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %5, pa;\n"
            "add.s64 ad, %1, 2;\nadd.s64 bd, %2, 2;\n"
            "@pe tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %5, pt;\n"
            "add.s64 ad, %1, 4;\nadd.s64 bd, %2, 4;\n"
            "@pe tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %5, pt;\n"
            "add.s64 ad, %1, 6;\nadd.s64 bd, %2, 6;\n"
            "@pe tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %5, pt;\n}\n" ::"r"(d),
            "l"(adesc), "l"(bdesc), "r"(acc0), "r"(issue), "n"(kIdesc)
            : "memory");
    // kMC: the commit arrives on the barrier at this offset in both CTAs of the cluster
    if constexpr (kMC)
        asm volatile(
            "{\n.reg .pred pe;\nsetp.ne.b32 pe, %1, 0;\n"
            "@pe tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %2;\n}\n" ::"r"(bar),
            "r"(issue), "h"(static_cast<uint16_t>(3))
            : "memory");
    else
        asm volatile(
            "{\n.reg .pred pe;\nsetp.ne.b32 pe, %1, 0;\n"
            "@pe tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n}\n" ::"r"(bar),
            "r"(issue)
            : "memory");
}

// ---- one kernel row of a 3x3 halo tile with resident weights ----
// The three taps (kh, 0..2) of a row: A from the halo buffer at the row's first
// tap (descriptor adesc; + 8 units, one 128-byte row, per tap), B from the
// stages of the three taps (bdesc, + kSU units per stage); four 16-deep MMAs per
// tap, twelve in one block from the issuing thread, no commit (resident weight
// stages are never released).  acc0: whether the first MMA accumulates.
template <uint32_t kIdesc, uint32_t kSU>
__device__ __forceinline__ void row3_f16(uint32_t d, uint64_t adesc, uint64_t bdesc, uint32_t acc0)
{
    asm volatile(
        "{\n.reg .pred pa, pt;\n.reg .b64 ad, bd, a1, b1;\n"
        "setp.ne.b32 pa, %3, 0;\nsetp.eq.b32 pt, 0, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %4, pa;\n"
        "add.s64 ad, %1, 2;\nadd.s64 bd, %2, 2;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 ad, %1, 4;\nadd.s64 bd, %2, 4;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 ad, %1, 6;\nadd.s64 bd, %2, 6;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 a1, %1, 8;\nadd.s64 b1, %2, %5;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], a1, b1, %4, pt;\n"
        "add.s64 ad, a1, 2;\nadd.s64 bd, b1, 2;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 ad, a1, 4;\nadd.s64 bd, b1, 4;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 ad, a1, 6;\nadd.s64 bd, b1, 6;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 a1, %1, 16;\nadd.s64 b1, b1, %5;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], a1, b1, %4, pt;\n"
        "add.s64 ad, a1, 2;\nadd.s64 bd, b1, 2;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 ad, a1, 4;\nadd.s64 bd, b1, 4;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 ad, a1, 6;\nadd.s64 bd, b1, 6;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], ad, bd, %4, pt;\n}\n" ::"r"(d),
        "l"(adesc), "l"(bdesc), "r"(acc0), "n"(kIdesc), "n"(static_cast<uint64_t>(kSU))
        : "memory");
}

// ---- one pipeline stage of bf16 MMAs over a CTA pair ----
// The four 16-deep cta_group::2 MMAs of a 64-wide stage (issued by the even CTA;
// descriptors advance by 32 bytes per MMA) and the commit that releases the
// stage in both CTAs (arrival multicast to the barrier at this offset in each),
// from one block executed by the issuing thread alone.  The separate per-MMA
// form took ~360 cycles per stage to issue on GB300 (clock stamps), against 512
// cycles of MMA work: the issue, not the tensor pipe, set the stage period.
template <uint32_t kIdesc>
__device__ __forceinline__ void stage_f16_pair(uint32_t d, uint64_t adesc, uint64_t bdesc, uint32_t acc0,
                                               uint32_t bar)
{
    asm volatile(
        "{\n.reg .pred pa, pt;\n.reg .b64 ad, bd;\n"
        "setp.ne.b32 pa, %3, 0;\nsetp.eq.b32 pt, 0, 0;\n"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %4, pa;\n"
        "add.s64 ad, %1, 2;\nadd.s64 bd, %2, 2;\n"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 ad, %1, 4;\nadd.s64 bd, %2, 4;\n"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], ad, bd, %4, pt;\n"
        "add.s64 ad, %1, 6;\nadd.s64 bd, %2, 6;\n"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], ad, bd, %4, pt;\n"
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%5], %6;\n}\n" ::"r"(d),
        "l"(adesc), "l"(bdesc), "r"(acc0), "n"(kIdesc), "r"(bar), "h"(static_cast<uint16_t>(3))
        : "memory");
}

// ---- cluster-pair helpers (CG = 2) ----
__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// shared::cluster address of the same shared variable in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t map_to_rank(uint32_t local, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
    return r;
}

__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr)
{
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// arrival on the even CTA's barrier that releases this thread's (and, through a
// preceding warp or CTA barrier, its peers') shared-memory writes: a release
// fence restricted to shared::cta accesses, then a relaxed arrive.  Measured on
// GB300 in the fused family's producer loop: ~950 cycles per stage for the
// cluster-scope release arrive above, a few hundred for this form.
__device__ __forceinline__ void mbar_arrive_remote_smem(uint32_t cluster_addr)
{
    asm volatile("fence.release.sync_restrict::shared::cta.cluster;" ::: "memory");
    asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// tcgen05.commit of the pair's MMAs, arriving on the barrier at this offset in both CTAs
__device__ __forceinline__ void mma_commit_pair(uint64_t *bar)
{
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
            tc::smem_u32(bar)),
        "h"(static_cast<uint16_t>(3))
        : "memory");
}

// TMA loads of either CTA of the pair completing on the even CTA's barrier
// (cluster address)
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const void *tmap, int x, int y, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, "
        "{%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// 2-D tile copy into the same shared-memory offset of both CTAs of a cluster of
// two, completing on the barrier at the same offset in each
__device__ __forceinline__ void tma_load_2d_mc(uint32_t dst, const void *tmap, int x, int y, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.multicast::cluster [%0], [%1, "
        "{%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(bar), "h"(static_cast<uint16_t>(3))
        : "memory");
}

__device__ __forceinline__ void tma_load_4d_pair(uint32_t dst, const void *tmap, int c0, int c1, int c2, int c3,
                                                 uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.tensor.4d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, "
        "{%2, %3, %4, %5}], [%6];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
        : "memory");
}

// Output epilogue of a CNN layer, on 32 consecutive fp32 accumulator values of
// one row at output channels col0..col0+31: y + bias[co] (when p.bias), then
// max(y, 0) (when p.relu).  Channels >= Cout get no bias (their columns are
// clipped by the store).
__device__ __forceinline__ void epilogue_math(uint32_t (&v)[32], const FwdParams &p, int col0)
{
    if (p.bias) {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            const int col = col0 + 4 * q;
            // Cout is a multiple of 4 and the bias 16-byte aligned: a float4 that
            // starts inside the row of biases lies wholly inside it
            const float4 b = col < p.Cout ? __ldg(reinterpret_cast<const float4 *>(p.bias + col))
                                          : make_float4(0.f, 0.f, 0.f, 0.f);
            v[4 * q] = __float_as_uint(__uint_as_float(v[4 * q]) + b.x);
            v[4 * q + 1] = __float_as_uint(__uint_as_float(v[4 * q + 1]) + b.y);
            v[4 * q + 2] = __float_as_uint(__uint_as_float(v[4 * q + 2]) + b.z);
            v[4 * q + 3] = __float_as_uint(__uint_as_float(v[4 * q + 3]) + b.w);
        }
    }
    if (p.relu) {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
            const float x = __uint_as_float(v[j]);
            v[j] = __float_as_uint(x > 0.f ? x : 0.f);
        }
    }
}

// two fp32 values (lo at the lower address) rounded to nearest even bf16
__device__ __forceinline__ uint32_t bf16x2_rn(uint32_t lo, uint32_t hi)
{
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(__uint_as_float(hi)), "f"(__uint_as_float(lo)));
    return r;
}

// byte offset of (row, 16-byte chunk) in a plane of 128-byte rows, 128-byte swizzle
__device__ __forceinline__ uint32_t sw_chunk(int row, int chunk)
{
    return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) * 16));
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c, uint32_t d)
{
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}
__device__ __forceinline__ void st_shared_v2(uint32_t addr, uint32_t a, uint32_t b)
{
    asm volatile("st.shared.v2.b32 [%0], {%1, %2};" ::"r"(addr), "r"(a), "r"(b) : "memory");
}

// the gathered fp32 activations x[0..3] of one 16-byte chunk of an A row, split
// into the operand planes (cci_common.cuh): the tf32 hi into plane 0 (at
// plane0), the bf16 pairs of x and lo(x) into plane 1 (at plane1), 8 bytes each
// at their places of the 128-byte-swizzled row
__device__ __forceinline__ void st_shared_x_split(uint32_t plane0, uint32_t plane1, int row, int chunk, uint4 v)
{
    const uint32_t x[4] = {v.x, v.y, v.z, v.w};
    uint32_t h[4];
    float l[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        h[e] = tf32_trunc(x[e]);
        l[e] = __uint_as_float(x[e]) - __uint_as_float(h[e]);
    }
    st_shared_v4(plane0 + sw_chunk(row, chunk), h[0], h[1], h[2], h[3]);
    const uint32_t half = static_cast<uint32_t>(chunk & 1) * 8;
    st_shared_v2(plane1 + sw_chunk(row, chunk >> 1) + half,
                 bf16x2_rn_sat(__uint_as_float(x[0]), __uint_as_float(x[1])),
                 bf16x2_rn_sat(__uint_as_float(x[2]), __uint_as_float(x[3])));
    st_shared_v2(plane1 + sw_chunk(row, 4 + (chunk >> 1)) + half, bf16x2_rn_sat(l[0], l[1]), bf16x2_rn_sat(l[2], l[3]));
}


// ---- expansion of packed weights into a B tile (PK) ----
// One producer thread builds an item: 8 consecutive B rows (output channels
// co0 + m0 .. + 7) x 8 consecutive reduction indices (one 16-byte chunk of each
// row).  Its inputs are the K-slot runs of the item's group(s) over those 8
// indices, loaded from the packed arrays ([r][slot]: values bf16, indices
// uint8) into registers.  Rows are built two indices (one 32-bit word: a bf16
// pair) at a time: for r-pair p and slot s, the pair's two values are ANDed with
// a mask that is 0xffff in each half whose index names the row, and ORed into
// the row's word.  The masks come from one packed f16x2 equality test per row:
// each index i of the pair becomes the f16 number with bits 0x3c00 | i (a key
// in [1, 2), distinct per index, exact), compared with the row's key; the test
// yields 0xffff per equal half.
namespace pk {

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel)
{
    uint32_t r;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
    return r;
}

// 0xffff in each half of a where it equals the same half of b (both f16x2)
__device__ __forceinline__ uint32_t eq_mask(uint32_t a, uint32_t b)
{
    uint32_t r;
    asm("set.eq.u32.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

// key of row jj in both halves
__device__ __forceinline__ constexpr uint32_t row_key(int jj) { return (0x3c00u | static_cast<uint32_t>(jj)) * 0x00010001u; }

// values of slot s at r = 2p (low half) and 2p + 1 (high half); vw holds the
// item's K-slot runs, v[r][s] at bf16 position r * K + s
template <int K>
__device__ __forceinline__ uint32_t val_pair(const uint32_t *vw, int p, int s)
{
    if constexpr (K == 1) {
        return vw[p];
    } else {
        const int e0 = 2 * p * K + s, e1 = (2 * p + 1) * K + s;  // bf16 positions
        return prmt(vw[e0 >> 1], vw[e1 >> 1], (e0 & 1 ? 0x32u : 0x10u) | (e1 & 1 ? 0x7600u : 0x5400u));
    }
}

// keys of the indices of slot s at r = 2p (low half) and 2p + 1 (high half):
// bytes (index, 0x3c, index, 0x3c)
template <int K>
__device__ __forceinline__ uint32_t key_pair(const uint32_t *iw, int p, int s)
{
    const int b0 = 2 * p * K + s, b1 = (2 * p + 1) * K + s;
    if ((b0 >> 2) == (b1 >> 2))
        return prmt(iw[b0 >> 2], 0x3c3c3c3cu, static_cast<uint32_t>((b0 & 3) | 0x40 | ((b1 & 3) << 8) | 0x4000));
    return (prmt(iw[b0 >> 2], iw[b1 >> 2], static_cast<uint32_t>((b0 & 3) | ((4 + (b1 & 3)) << 8))) & 0x00ff00ffu) |
           0x3c003c00u;
}

// adds one group's K slots to rows J0 .. J1 - 1 of the item: a slot of index i
// goes to row i + off (off: 4 for the second group of a G = 4 item, -j0 for
// G >= 16, whose items cover rows j0 .. j0 + 7 of their group; slots whose row
// lies outside add nothing).  INIT: these rows start from this group's
// contributions.
template <int K, int J0, int J1, bool INIT>
__device__ __forceinline__ void expand_group(uint32_t (&out)[8][4], const uint32_t *vw, const uint32_t *iw, int off)
{
    const uint32_t kadd = static_cast<uint32_t>(off) * 0x00010001u;  // off + 0x3c00 >= 0 in each half: no borrow
#pragma unroll
    for (int pr = 0; pr < 4; ++pr) {
#pragma unroll
        for (int s = 0; s < K; ++s) {
            const uint32_t v = val_pair<K>(vw, pr, s);
            const uint32_t key = key_pair<K>(iw, pr, s) + kadd;
#pragma unroll
            for (int jj = J0; jj < J1; ++jj) {
                const uint32_t m = eq_mask(key, row_key(jj));
                if (INIT && s == 0)
                    out[jj][pr] = v & m;
                else
                    out[jj][pr] |= v & m;
            }
        }
    }
}

// true if an index set of the group at one of the item's first nr reduction
// indices is not strictly increasing or has an index >= G (cci_pack never
// writes such sets)
template <int K>
__device__ __forceinline__ bool bad_sets(const uint32_t *iw, int G, int nr)
{
    bool bad = false;
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        if (r >= nr) break;
        int prev = -1;
#pragma unroll
        for (int s = 0; s < K; ++s) {
            const int b = r * K + s;
            const int j = static_cast<int>((iw[b >> 2] >> (8 * (b & 3))) & 0xffu);
            bad |= j >= G || j <= prev;
            prev = j;
        }
    }
    return bad;
}

// the K-slot runs of an item's group(s) at its 8 reduction indices, in
// registers: NG groups (2 for G = 4, whose items span two groups), per group
// 4K words of values (v[r][s] at bf16 position r*K + s) and 2K words of indices
template <int K>
struct Runs {
    static constexpr int NG = K <= 2 ? 2 : 1;
    uint32_t v[NG][4 * K];
    uint32_t i[NG][2 * K];
};

// global loads of one group's runs at reduction indices r .. r + 7: 16 K bytes
// of values and 8 K bytes of indices from offset (g*R + r)*K of the packed
// arrays (16-byte aligned: R % 8 == 0, r % 8 == 0); zeros for a group past the
// last one or indices past R (R % 8 == 0, so a chunk is wholly inside or out)
template <int K>
__device__ __forceinline__ void load_group(uint32_t (&v)[4 * K], uint32_t (&iw)[2 * K], const uint16_t *V,
                                           const uint8_t *I, int64_t g, int64_t groups, int64_t r, int64_t R)
{
    if (g < groups && r < R) {
        const int64_t off = (g * R + r) * K;
        const uint4 *pv = reinterpret_cast<const uint4 *>(V + off);
#pragma unroll
        for (int q = 0; q < K; ++q) {
            const uint4 x = __ldg(pv + q);
            v[4 * q] = x.x;
            v[4 * q + 1] = x.y;
            v[4 * q + 2] = x.z;
            v[4 * q + 3] = x.w;
        }
        if constexpr (K == 1) {
            const uint2 x = __ldg(reinterpret_cast<const uint2 *>(I + off));
            iw[0] = x.x;
            iw[1] = x.y;
        } else {
            const uint4 *pi = reinterpret_cast<const uint4 *>(I + off);
#pragma unroll
            for (int q = 0; q < K / 2; ++q) {
                const uint4 x = __ldg(pi + q);
                iw[4 * q] = x.x;
                iw[4 * q + 1] = x.y;
                iw[4 * q + 2] = x.z;
                iw[4 * q + 3] = x.w;
            }
        }
    } else {
#pragma unroll
        for (int q = 0; q < 4 * K; ++q) v[q] = 0u;
#pragma unroll
        for (int q = 0; q < 2 * K; ++q) iw[q] = 0u;  // index 0 with value 0: adds nothing
    }
}

// the runs of the item whose first row is in group g (rows of groups g and g + 1
// for G = 4) at reduction indices r .. r + 7
template <int K>
__device__ __forceinline__ void load_item(Runs<K> &run, const FwdParams &p, int64_t g, int64_t r, int64_t groups)
{
    const uint16_t *V = static_cast<const uint16_t *>(p.values);
    if constexpr (Runs<K>::NG == 2) {
        if (p.G == 4) {
            load_group<K>(run.v[0], run.i[0], V, p.idx, g, groups, r, p.R);
            load_group<K>(run.v[1], run.i[1], V, p.idx, g + 1, groups, r, p.R);
            return;
        }
    }
    load_group<K>(run.v[0], run.i[0], V, p.idx, g, groups, r, p.R);
}

// the item's 8 rows of 8 bf16 (4 words each) from its runs (group g, first row
// j0 of the group); chk: check the index sets of its group(s) at the first nr
// indices (bad set on a bad one)
template <int K>
__device__ __forceinline__ void expand_item(uint32_t (&out)[8][4], const Runs<K> &run, int G, int64_t g, int j0,
                                            int64_t groups, int nr, bool chk, bool &bad)
{
    if constexpr (Runs<K>::NG == 2) {
        if (G == 4) {
            if (chk && g < groups) bad |= bad_sets<K>(run.i[0], G, nr);
            if (chk && g + 1 < groups) bad |= bad_sets<K>(run.i[1], G, nr);
            expand_group<K, 0, 4, true>(out, run.v[0], run.i[0], 0);
            expand_group<K, 4, 8, true>(out, run.v[1], run.i[1], 4);
            return;
        }
    }
    if (chk && j0 == 0 && g < groups) bad |= bad_sets<K>(run.i[0], G, nr);
    expand_group<K, 0, 8, true>(out, run.v[0], run.i[0], -j0);  // G = 8: j0 = 0
}

}  // namespace pk

// (box along q, box along p, batch box) of M tile mt
struct BoxIdx {
    int qb, pb;
    int64_t bb;
};
__device__ __forceinline__ BoxIdx box_of(int64_t mt, const ConvBox &box)
{
    BoxIdx i;
    i.qb = static_cast<int>(mt % box.nQ);
    const int64_t t = mt / box.nQ;
    i.pb = static_cast<int>(t % box.nP);
    i.bb = t / box.nP;
    return i;
}

// PK: tmB0 / tmB1 are the maps of the packed values and indices (2-D over
// [Cout/G][R*K]); otherwise the maps of the workspace planes
template <bool TF32, int ASRC, int BN, int CG, int EPI, bool PK = false, bool MC = false>
__global__ void __launch_bounds__(Cfg<TF32, ASRC, BN, CG, EPI, PK, MC>::kThreads, 1)
    gemm_ws_kernel(FwdParams p, const __grid_constant__ AMaps tmA, const __grid_constant__ CUtensorMap tmB0,
                   const __grid_constant__ CUtensorMap tmB1, const __grid_constant__ CUtensorMap tmY, ConvBox box,
                   int64_t n_ct, int64_t n_tiles)
{
    using C = Cfg<TF32, ASRC, BN, CG, EPI, PK, MC>;
    constexpr int kM = C::kM, kN = C::kN, kKS = C::kKS, kStages = C::kStages;
    constexpr int kLag = 2;  // bf16 gather: stages in flight before a producer's arrive
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const uint32_t raw = tc::smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    const uint32_t hbuf = base + kStages * C::kStage;  // halo ring (kAHalo: box.nh buffers)
    const uint32_t hbytes = static_cast<uint32_t>(box.hrows) * 128u;
    const uint32_t hring = C::kHalo ? static_cast<uint32_t>(box.nh) * hbytes : 0u;
    const uint32_t ybuf = hbuf + hring;  // output staging buffers, two per epilogue group
    tc::Smem *S = reinterpret_cast<tc::Smem *>(smem_raw + (base - raw) + kStages * C::kStage + hring +
                                               C::kYBufs * C::kYBuf);
    const int taps = p.KH * p.KW;  // kAHalo: stages run chunk by chunk, the taps of a chunk in turn
    volatile int *abort = &S->abort;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nks = static_cast<int>((p.R + kKS - 1) / kKS);
    const uint32_t crank = C::kPairUnits ? cluster_rank() : 0u;  // CG = 2: 0 issues the pair's MMAs
    // work units: tiles (CG = 1) or pair tiles of 2 x 128 rows (CG = 2), strided over
    // the CTAs (CG = 1) or the CTA pairs (CG = 2)
    const int64_t u0 = C::kPairUnits ? blockIdx.x / 2 : blockIdx.x;
    const int64_t ustep = C::kPairUnits ? gridDim.x / 2 : gridDim.x;
    // unit u -> (M tile, N tile): one 64-bit division, the remainder by multiply-subtract
    auto split_unit = [&](int64_t u, int64_t &mt, int64_t &ct) {
        const int64_t q = u / n_ct;
        ct = u - q * n_ct;
        mt = C::kPairUnits ? 2 * q + crank : q;
    };

    if (tid == 0) {
        // full[s]: the copy issuer's expect_tx arrival (none for PK halo stages) and
        // PK: one arrival per producer warp of the stage's group in each CTA of the
        // pair (after the warp's writes), else 128 producer arrivals when the
        // producers fill the stage
        const uint32_t full_count = PK ? (C::kHalo ? 0u : 1u) + 4 * CG : (C::kATma ? 1u : 129u);
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(&S->full[s], full_count);
            tc::mbar_init(&S->empty[s], MC ? 2 : 1);  // MC: released by both CTAs' MMAs
            tc::mbar_init(&S->aux[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            tc::mbar_init(&S->tmem_full[a], 1);
            tc::mbar_init(&S->tmem_empty[a], 128 * CG);
        }
        tc::mbar_init(&S->drain, 1);
        for (int h = 0; h < tc::kMaxHalo; ++h) {
            tc::mbar_init(&S->hfull[h], 1);
            tc::mbar_init(&S->hempty[h], 1);
        }
        S->abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (ASRC == kA4d && box.rows < kM) {
        // rows past the box are never copied: keep them zero for the MMAs
        for (uint32_t o = static_cast<uint32_t>(tid) * 16; o < static_cast<uint32_t>(kStages * C::kStage);
             o += C::kThreads * 16)
            tc::st_shared_v4_zero(base + o);
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 8) {
        if constexpr (CG == 2) {  // one warp of each CTA of the pair, collectively
            asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                             tc::smem_u32(&S->tmem_base)),
                         "r"(C::kTmemCols)
                         : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
        } else {
            asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                             tc::smem_u32(&S->tmem_base)),
                         "r"(C::kTmemCols)
                         : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
        }
    }
    if (tid == 288) {
        if constexpr (ASRC == kA2d) tc::tma_prefetch_desc(&tmA.m[0]);
        if constexpr (ASRC == kA4d)
            for (int i = 0; i < p.sh * p.sw; ++i) tc::tma_prefetch_desc(&tmA.m[i]);
        if constexpr (ASRC == kAHalo) tc::tma_prefetch_desc(&tmA.m[0]);
        if constexpr (!PK) tc::tma_prefetch_desc(&tmB0);
        if constexpr (C::kBPlanes > 1) tc::tma_prefetch_desc(&tmB1);
        tc::tma_prefetch_desc(&tmY);
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    // the pair's barriers are initialised before either CTA signals the other's
    if constexpr (C::kPairUnits) cluster_sync();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = S->tmem_base;
    // launched as a programmatic dependent of the decompression: everything above
    // overlaps its tail; the workspace (and anything else in memory) is read only
    // after that grid has completed and its writes are visible
    asm volatile("griddepcontrol.wait;" ::: "memory");

    if (warp >= 9 && warp < 9 + C::kIssuers) {
        // ------------------------------------------------------------ TMA issuers
        // bytes of one stage's copies: rows x the indices copied per stage (fewer than
        // the stage depth only for bf16 products of fewer than 64 reduction indices,
        // which run in the two-group short-tile form)
        const uint32_t erow = static_cast<uint32_t>(EPI == 2 ? p.kin : kKS) * (TF32 ? 4u : 2u);  // bytes per row
        const uint32_t a_bytes = (ASRC == kA4d ? static_cast<uint32_t>(box.rows) : static_cast<uint32_t>(kM)) * erow;
        const uint32_t b_bytes = static_cast<uint32_t>(C::kBPlanes * C::kBRows) * erow;
        const int cpt = static_cast<int>(p.Cin / kKS);  // stages per tap (kA4d)
        const uint32_t halo_bytes =
            static_cast<uint32_t>((box.QB + p.KW - 1) * (box.PB + p.KH - 1)) * 128u;  // kAHalo
        // kAHalo: warp 9 copies the halos, as far ahead as the halo ring allows;
        // the other issuer warps copy the weight stages in turn
        const int issuer = warp - (C::kHalo ? 10 : 9);
        constexpr int kBIssuers = C::kHalo ? C::kIssuers - 1 : C::kIssuers;
        int it = 0;
        bool ok = true;
        if (C::kHalo && warp == 9) {
            int hc = 0;
            const int chunks = nks / taps;
            for (int64_t u = u0; u < n_tiles && ok; u += ustep) {
                int64_t mt, ct;
                split_unit(u, mt, ct);
                const BoxIdx bi = box_of(mt, box);
                for (int c = 0; c < chunks && ok; ++c, ++hc) {
                    // buffer hb is free once the MMAs of chunk hc - nh completed; this
                    // warp waited for chunk hc - 1 - nh before, so the phase cannot alias
                    const int hb = hc % box.nh;
                    if (hc >= box.nh) ok = tc::mbar_wait(&S->hempty[hb], ((hc / box.nh) - 1) & 1, abort, p.status);
                    if (!ok) break;
                    if (lane == 0) {
                        if constexpr (CG == 2) {
                            // each CTA's halo (its own M tile) completes on the even CTA's
                            // barrier, which expects both
                            if (crank == 0) tc::mbar_arrive_expect_tx(&S->hfull[hb], 2 * halo_bytes);
                            tma_load_4d_pair(hbuf + hb * hbytes, &tmA.m[0], c * 64, -p.pw, bi.pb * box.PB - p.ph,
                                             static_cast<int>(bi.bb), map_to_rank(tc::smem_u32(&S->hfull[hb]), 0));
                        } else {
                            tc::mbar_arrive_expect_tx(&S->hfull[hb], halo_bytes);
                            tc::tma_load_4d(hbuf + hb * hbytes, &tmA.m[0], c * 64, -p.pw, bi.pb * box.PB - p.ph,
                                            static_cast<int>(bi.bb), &S->hfull[hb]);
                        }
                    }
                    __syncwarp();
                }
            }
        } else if (!(PK && C::kHalo))  // PK halo stages hold only the producers' weight tiles
        for (int64_t u = u0; u < n_tiles && ok; u += ustep) {
            int64_t mt, ct;
            split_unit(u, mt, ct);
            const int64_t co0 = ct * kN + (CG == 2 ? crank * C::kBRows : 0);  // this CTA's B rows
            BoxIdx bi{0, 0, 0};
            if constexpr (ASRC == kA4d || ASRC == kAHalo) bi = box_of(mt, box);
            // resident weights (halo copies): only the first tile's stages are copied
            if (C::kHalo && box.resident && it >= nks) break;
            for (int ks = 0; ks < nks && ok; ++ks, ++it) {
                if (it % kBIssuers != issuer) continue;
                const int s = it % kStages;
                if (it >= kStages) ok = tc::mbar_wait(&S->empty[s], ((it / kStages) - 1) & 1, abort, p.status);
                if (!ok) break;
                if constexpr (ASRC == kAHalo) {
                    const int c = ks / taps, t = ks - c * taps;  // stages: chunk by chunk, taps in turn
                    if (lane == 0) {
                        const int x = static_cast<int>(t * p.Cin) + c * 64;
                        if constexpr (CG == 2) {  // this CTA's half of the rows, on the even CTA's barrier
                            if (crank == 0) tc::mbar_arrive_expect_tx(&S->full[s], 2 * C::kBBytes);
                            tma_load_2d_pair(base + s * C::kStage, &tmB0, x, static_cast<int>(co0),
                                             map_to_rank(tc::smem_u32(&S->full[s]), 0));
                        } else {
                            tc::mbar_arrive_expect_tx(&S->full[s], C::kBBytes);
                            tc::tma_load_2d(base + s * C::kStage, &tmB0, x, static_cast<int>(ct * kN), &S->full[s]);
                        }
                    }
                    __syncwarp();
                    continue;
                }
                if (lane == 0 && CG == 2) {
                    // both CTAs' copies complete on the even CTA's full barrier, which
                    // expects the bytes of the pair (PK: the activations only; each
                    // CTA's packed runs land on its own aux barrier)
                    const uint32_t st = base + s * C::kStage;
                    const uint32_t bst = st + C::kAPlane;
                    const uint32_t fb = map_to_rank(tc::smem_u32(&S->full[s]), 0);
                    if constexpr (PK) {
                        if (crank == 0) tc::mbar_arrive_expect_tx(&S->full[s], 2 * a_bytes);
                    } else {
                        if (crank == 0) tc::mbar_arrive_expect_tx(&S->full[s], 2 * (C::kBBytes + a_bytes));
                        tma_load_2d_pair(bst, &tmB0, ks * kKS, static_cast<int>(co0), fb);
                    }
                    if constexpr (ASRC == kA2d) {
                        tma_load_2d_pair(st, &tmA.m[0], ks * kKS, static_cast<int>(mt * kM), fb);
                    } else {
                        const int tap = ks / cpt;
                        const int ci0 = (ks - tap * cpt) * kKS;
                        const int kh = tap / p.KW, kw = tap - (tap / p.KW) * p.KW;
                        const int ah = kh - p.ph, aw = kw - p.pw;
                        const int rh = ((ah % p.sh) + p.sh) % p.sh, rw = ((aw % p.sw) + p.sw) % p.sw;
                        const int dh = (ah - rh) / p.sh, dw = (aw - rw) / p.sw;
                        tma_load_4d_pair(st, &tmA.m[rh * p.sw + rw], ci0, bi.qb * box.QB + dw,
                                         bi.pb * box.PB + dh, static_cast<int>(bi.bb * box.BB), fb);
                    }
                } else if (lane == 0) {
                    const uint32_t st = base + s * C::kStage;
                    const uint32_t bst = st + C::kBOff;
                    // the activation copy completes on aux (raw fp32, split afterwards) or full
                    uint64_t *abar = C::kARaw ? &S->aux[s] : &S->full[s];
                    if constexpr (C::kARaw) tc::mbar_arrive_expect_tx(abar, a_bytes);
                    if constexpr (PK) {
                        tc::mbar_arrive_expect_tx(&S->full[s], a_bytes);
                    } else {
                        tc::mbar_arrive_expect_tx(&S->full[s], b_bytes + (C::kATma ? a_bytes : 0u));
                        if constexpr (MC) {
                            // this CTA's half of the B rows into both CTAs (the same offsets);
                            // each CTA's full barrier expects the whole tile
                            const uint32_t half = crank * (C::kBPlane / 2);
                            const int y = static_cast<int>(co0) + static_cast<int>(crank) * (kN / 2);
                            tma_load_2d_mc(bst + half, &tmB0, ks * kKS, y, tc::smem_u32(&S->full[s]));
                            if constexpr (C::kBPlanes > 1)
                                tma_load_2d_mc(bst + C::kBPlane + half, &tmB1, ks * 64, y, tc::smem_u32(&S->full[s]));
                        } else {
                            tc::tma_load_2d(bst, &tmB0, ks * kKS, static_cast<int>(co0), &S->full[s]);
                            if constexpr (C::kBPlanes > 1)  // fp32 plane 1: 64 bf16 per stage
                                tc::tma_load_2d(bst + C::kBPlane, &tmB1, ks * 64, static_cast<int>(co0), &S->full[s]);
                        }
                    }
                    if constexpr (ASRC == kA2d) {
                        tc::tma_load_2d(st, &tmA.m[0], ks * kKS, static_cast<int>(mt * kM), abar);
                    } else if constexpr (ASRC == kA4d) {
                        const int tap = ks / cpt;
                        const int ci0 = (ks - tap * cpt) * kKS;
                        const int kh = tap / p.KW, kw = tap - (tap / p.KW) * p.KW;
                        // input row h = p_out * sh + ah lies on lattice rh at h' = p_out + dh
                        const int ah = kh - p.ph, aw = kw - p.pw;
                        const int rh = ((ah % p.sh) + p.sh) % p.sh, rw = ((aw % p.sw) + p.sw) % p.sw;
                        const int dh = (ah - rh) / p.sh, dw = (aw - rw) / p.sw;
                        tc::tma_load_4d(st, &tmA.m[rh * p.sw + rw], ci0, bi.qb * box.QB + dw, bi.pb * box.PB + dh,
                                        static_cast<int>(bi.bb * box.BB), abar);
                    }
                }
                __syncwarp();
            }
        }
    } else if (PK && ((warp >= 4 && warp < 8) || warp >= 9 + C::kIssuers)) {
        // ------------------------------------------------------------ weight producers (PK)
        // two groups of four warps (4-7 and the four after the issuers) take the
        // stages in turn: group q builds the stages it with it % 2 == q, so each
        // group has two MMA stages of time per tile it builds.  Thread pt of a
        // group builds item pt of each of its stages: rows 8 (pt / 8) .. + 7 of
        // this CTA's B tile, reduction indices 8 (pt % 8) .. + 7 of the stage.  Its
        // runs are loaded NB of its stages ahead into a ring of NB register sets (a
        // set is refilled right after it is expanded), expanded into rows while the
        // stage may still be in use, and stored once the stage's MMAs released it;
        // then each warp releases its writes to the stage's full barrier (pair: the
        // even CTA's).
        const int q = warp >= 8 ? 1 : 0;
        const int pt = tid - (q ? 32 * (9 + C::kIssuers) : 128);
        const int m0 = (pt >> 3) * 8, c = pt & 7;
        const bool active = m0 < C::kBRows;
        const int64_t groups = p.Cout / p.G;
        const int lg = 31 - __clz(p.G);  // G is a power of two
        const uint32_t full_remote = CG == 2 ? map_to_rank(tc::smem_u32(&S->full[0]), 0) : 0u;
        bool bad = false;
        // a stage of this CTA, in the MMAs' order, and the item's place in it: the
        // output channel of its first row, its group, the reduction index of its
        // first column, whether its tile checks index sets (the first M tile, or
        // pair, of each N tile).  Advanced stage by stage without division (one
        // per tile).
        struct Cursor {
            int64_t u, co, g, r;
            int ks, t, ch, j0;
            bool chk;
        };
        auto tile_start = [&](Cursor &cu) {
            if (cu.u >= n_tiles) return;
            int64_t mt, ct;
            split_unit(cu.u, mt, ct);
            cu.co = ct * kN + crank * C::kBRows + m0;
            cu.g = cu.co >> lg;
            cu.j0 = static_cast<int>(cu.co & (p.G - 1));
            cu.chk = mt < CG;
            cu.ks = cu.t = cu.ch = 0;
            cu.r = 8 * c;
        };
        auto advance = [&](Cursor &cu) {
            if (++cu.ks == nks) {
                cu.u += ustep;
                tile_start(cu);
                return;
            }
            if constexpr (ASRC == kAHalo) {  // stages chunk by chunk, the taps of a chunk in turn
                if (++cu.t == taps) {
                    cu.t = 0;
                    ++cu.ch;
                }
                cu.r = static_cast<int64_t>(cu.t) * p.Cin + cu.ch * 64 + 8 * c;
            } else {
                cu.r += 64;
            }
        };
        auto run_k = [&](auto kc) {
            constexpr int K = decltype(kc)::value;
            constexpr int NB = K <= 4 ? 2 : 1;
            pk::Runs<K> ring[NB];
            Cursor cur{u0, 0, 0, 0, 0, 0, 0, 0, false};  // the stage being built
            tile_start(cur);
            if (q) advance(cur);  // group 1 starts at the second stage
            Cursor pre = cur;     // the stage whose runs are loaded next (NB of this group's ahead)
            auto load = [&](pk::Runs<K> &rg) {
                if (active && pre.u < n_tiles) pk::load_item<K>(rg, p, pre.g, pre.r, groups);
                advance(pre);
                advance(pre);
            };
#pragma unroll
            for (int b = 0; b < NB; ++b) load(ring[b]);
            bool ok = true;
            int s = q;     // stage of the ring
            int pass = 0;  // passes over the ring completed before this stage
            while (ok && cur.u < n_tiles) {
#pragma unroll
                for (int b = 0; b < NB; ++b) {
                    if (!ok || cur.u >= n_tiles) break;
                    uint32_t out[8][4];
                    if (active) {
                        const int64_t left = p.R - cur.r;
                        const int nr = left <= 0 ? 0 : (left >= 8 ? 8 : static_cast<int>(left));
                        pk::expand_item<K>(out, ring[b], p.G, cur.g, cur.j0, groups, nr, cur.chk, bad);
                    }
                    load(ring[b]);
                    if (pass > 0) ok = tc::mbar_wait(&S->empty[s], (pass - 1) & 1, abort, p.status);
                    if (ok && active) {
                        const uint32_t bst = base + s * C::kStage + C::kBOff;
#pragma unroll
                        for (int jj = 0; jj < 8; ++jj)
                            st_shared_v4(bst + sw_chunk(m0 + jj, c), out[jj][0], out[jj][1], out[jj][2], out[jj][3]);
                    }
                    // the warp's writes are visible to the MMAs (async proxy) once its
                    // lane 0 arrives after all of them (pair: on the even CTA's barrier)
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    __syncwarp();
                    ok = __all_sync(0xffffffffu, ok);
                    if (!ok) break;
                    if (lane == 0) {
                        if (CG == 2 && crank != 0)
                            mbar_arrive_remote_smem(full_remote + static_cast<uint32_t>(s * sizeof(uint64_t)));
                        else
                            tc::mbar_arrive(&S->full[s]);
                    }
                    advance(cur);
                    advance(cur);
                    s += 2;
                    if (s >= kStages) {
                        s -= kStages;
                        ++pass;
                    }
                }
            }
        };
        switch (p.K) {
            case 1: run_k(std::integral_constant<int, 1>{}); break;
            case 2: run_k(std::integral_constant<int, 2>{}); break;
            case 4: run_k(std::integral_constant<int, 4>{}); break;
            default: run_k(std::integral_constant<int, 8>{}); break;
        }
        if (bad) report(p.status, CCI_ERR_INDEX);
    } else if (warp >= 4 && warp < 8 && C::kEG == 1) {
        // ------------------------------------------------------------ producers
        const int pt = tid - 128;
        const int chunk = pt & 7;  // 16-byte chunk of every activation row this thread handles
        const int rowb = pt >> 3;  // rows rowb + 16 i
        int it = 0;
        bool ok = true;
        constexpr bool kRegs = TF32 && ASRC == kAGather;  // fp32 gather through registers
        // fp32 gather: activation chunks of the next two stages, in registers
        uint4 xa[kRegs ? 8 : 1], xb[kRegs ? 8 : 1], xc[kRegs ? 8 : 1];
        ColumnSite xsite[kRegs ? 8 : 1];  // column sites of the tile being prefetched
        int64_t xsite_tile = -1;
        auto load_x = [&](uint4 (&dst)[kRegs ? 8 : 1], int64_t tile, int ks) {
            if constexpr (kRegs) {
#pragma unroll
                for (int i = 0; i < 8; ++i) dst[i] = make_uint4(0, 0, 0, 0);
                if (tile >= n_tiles || ks >= nks) return;
                const int64_t n0 = (tile / n_ct) * kM;
                if (tile != xsite_tile) {
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const int64_t n = n0 + rowb + 16 * i;
                        xsite[i] = n < p.N ? column_site(p, n) : ColumnSite{-1, 0, 0};
                    }
                    xsite_tile = tile;
                }
                const int64_t r = static_cast<int64_t>(ks) * kKS + chunk * 4;
                if (r >= p.R) return;
                int kh = 0, kw = 0;
                int64_t ci = r;
                if (p.is_conv) {
                    const int tap = static_cast<int>(r / p.Cin);
                    ci = r - static_cast<int64_t>(tap) * p.Cin;
                    kh = tap / p.KW;
                    kw = tap - kh * p.KW;
                }
                const float *X = static_cast<const float *>(p.X);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    if (xsite[i].img < 0) continue;  // column past N
                    int64_t off = xsite[i].img + r;
                    if (p.is_conv) {
                        const int h = xsite[i].hb + kh, w = xsite[i].wb + kw;
                        if (h < 0 || h >= p.H || w < 0 || w >= p.W) continue;
                        off = xsite[i].img + (static_cast<int64_t>(h) * p.W + w) * p.Cin + ci;
                    }
                    dst[i] = __ldg(reinterpret_cast<const uint4 *>(X + off));
                }
            }
        };
        // (tile, ks) of the stage after (tile, ks)
        auto advance = [&](int64_t &tile, int &ks) {
            if (++ks == nks) {
                ks = 0;
                tile += gridDim.x;
            }
        };
        int64_t t2 = blockIdx.x;
        int k2 = 0;
        if constexpr (kRegs) {
            load_x(xa, t2, k2);
            advance(t2, k2);
            load_x(xb, t2, k2);
            advance(t2, k2);
        }
        if constexpr (!C::kATma) {
            // the same work units, in the same order, as the TMA issuers and the MMAs
            for (int64_t tile = u0; tile < n_tiles && ok; tile += ustep) {
                const int64_t n0 = (tile / n_ct) * kM;
                ColumnSite site[8];
                bool colok[8];
                if constexpr (!TF32) {
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const int64_t n = n0 + rowb + 16 * i;
                        colok[i] = n < p.N;
                        site[i] = colok[i] ? column_site(p, n) : ColumnSite{0, 0, 0};
                    }
                }
                for (int ks = 0; ks < nks && ok; ++ks, ++it) {
                    const int s = it % kStages;
                    if constexpr (kRegs) load_x(xc, t2, k2);  // two stages ahead
                    // gather / register modes write the stage themselves: wait until it is
                    // free; the split mode waits for its raw tile (copied after the stage
                    // was freed) instead
                    if (!C::kARaw && it >= kStages)
                        ok = tc::mbar_wait(&S->empty[s], ((it / kStages) - 1) & 1, abort, p.status);
                    if (!ok) break;
                    const uint32_t st = base + s * C::kStage;
                    if constexpr (!TF32) {
                        const uint16_t *X = static_cast<const uint16_t *>(p.X);
                        const int64_t r = static_cast<int64_t>(ks) * kKS + chunk * 8;
                        const bool rok = r < p.R;
                        int kh = 0, kw = 0;
                        int64_t ci = r;
                        if (p.is_conv && rok) {
                            const int tap = static_cast<int>(r / p.Cin);
                            ci = r - static_cast<int64_t>(tap) * p.Cin;
                            kh = tap / p.KW;
                            kw = tap - kh * p.KW;
                        }
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            bool valid = colok[i] && rok;
                            const uint16_t *src = X;
                            if (valid) {
                                if (!p.is_conv) {
                                    src = X + site[i].img + r;
                                } else {
                                    const int h = site[i].hb + kh, w = site[i].wb + kw;
                                    valid = h >= 0 && h < p.H && w >= 0 && w < p.W;
                                    if (valid)
                                        src = X + site[i].img + (static_cast<int64_t>(h) * p.W + w) * p.Cin + ci;
                                }
                            }
                            tc::cp_async16(st + sw_chunk(rowb + 16 * i, chunk), src, valid);
                        }
                        asm volatile("cp.async.commit_group;" ::: "memory");
                        if (it >= kLag) {
                            asm volatile("cp.async.wait_group %0;" ::"n"(kLag) : "memory");
                            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                            tc::mbar_arrive(&S->full[(it - kLag) % kStages]);
                        }
                    } else if constexpr (C::kARaw) {
                        // the raw fp32 tile landed: row m = pt, split in registers (the
                        // operand planes of cci_common.cuh: hi(x) as tf32, then the bf16
                        // pairs of x and lo(x)) and written to this stage's 64 A columns
                        // of tensor memory (lane m; warp 4 + q owns lanes 32q..32q+31)
                        ok = tc::mbar_wait(&S->aux[s], (it / kStages) & 1, abort, p.status);
                        ok = __all_sync(0xffffffffu, ok);
                        if (!ok) break;
                        uint32_t hv[32], bv[32];
#pragma unroll
                        for (int q = 0; q < 8; ++q) {
                            uint4 v;
                            asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                                         : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                                         : "r"(st + sw_chunk(pt, q))
                                         : "memory");
                            const uint32_t x[4] = {v.x, v.y, v.z, v.w};
                            float l[4];
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                hv[4 * q + e] = tf32_trunc(x[e]);
                                l[e] = __uint_as_float(x[e]) - __uint_as_float(hv[4 * q + e]);
                            }
                            bv[2 * q] = bf16x2_rn_sat(__uint_as_float(x[0]), __uint_as_float(x[1]));
                            bv[2 * q + 1] = bf16x2_rn_sat(__uint_as_float(x[2]), __uint_as_float(x[3]));
                            bv[16 + 2 * q] = bf16x2_rn_sat(l[0], l[1]);
                            bv[16 + 2 * q + 1] = bf16x2_rn_sat(l[2], l[3]);
                        }
                        const uint32_t ta = tmem + (static_cast<uint32_t>((warp - 4) * 32) << 16) +
                                            static_cast<uint32_t>(C::kAColBase + s * 64);
                        tc::tmem_st32(ta, hv);
                        tc::tmem_st32(ta + 32, bv);
                        asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
                        asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                        tc::mbar_arrive(&S->full[s]);
                    } else {
#pragma unroll
                        for (int i = 0; i < 8; ++i) st_shared_x_split(st, st + C::kAPlane, rowb + 16 * i, chunk, xa[i]);
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                        tc::mbar_arrive(&S->full[s]);
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            xa[i] = xb[i];
                            xb[i] = xc[i];
                        }
                        advance(t2, k2);
                    }
                }
            }
            if constexpr (!TF32) {
                asm volatile("cp.async.wait_group 0;" ::: "memory");
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                for (int q = (it >= kLag ? it - kLag : 0); q < it; ++q) tc::mbar_arrive(&S->full[q % kStages]);
            }
        }
    } else if (warp == 8) {
        // ------------------------------------------------------------ MMA issuer
        // (CG = 2: the even CTA issues for the pair; the odd CTA only waits for
        // the drain)
        int it = 0, t = 0;
        bool ok = CG == 1 || crank == 0;
        const int hchunks = ASRC == kAHalo ? nks / taps : 0;
        const uint64_t hdesc0 = tc::sw128_desc(hbuf), bdesc0 = tc::sw128_desc(base);
        const uint32_t empty0 = tc::smem_u32(&S->empty[0]);
        const uint32_t issue = lane == 0 ? 1u : 0u;  // the lane that issues (a predicate in the stage block)
        auto commit = [&](uint64_t *bar) {
            if constexpr (CG == 2)
                mma_commit_pair(bar);
            else
                tc::mma_commit(bar);
        };
        if constexpr (C::kARaw) {
            // one thread runs the whole issue loop: no per-stage divergence or warp
            // reconvergence between the stages' MMAs (the gaps between stages, not
            // the MMAs, bounded this product)
            if (lane == 0) {
                for (int64_t u = u0; u < n_tiles && ok; u += ustep, ++t) {
                    const int acc = t & 1;
                    if (t >= 2) ok = tc::mbar_wait(&S->tmem_empty[acc], ((t / 2) - 1) & 1, abort, p.status);
                    if (!ok) break;
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint32_t d = tmem + static_cast<uint32_t>(acc * kN);
                    for (int ks = 0; ks < nks; ++ks, ++it) {
                        const int s = it % kStages;
                        ok = tc::mbar_wait(&S->full[s], (it / kStages) & 1, abort, p.status);
                        if (!ok) break;
                        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                        stage_tf32_split<C::kIdesc, C::kIdescB, (C::kBPlane >> 4), MC>(
                            d, tmem + static_cast<uint32_t>(C::kAColBase + s * 64),
                            bdesc0 + static_cast<uint64_t>(s) * (C::kStage >> 4) + (C::kBOff >> 4), ks > 0 ? 1u : 0u,
                            1u, empty0 + 8u * s);
                    }
                    if (ok) commit(&S->tmem_full[acc]);
                }
            }
            ok = false;  // the generic loop below is not entered
        }
        if constexpr (!TF32 && ASRC != kAHalo) {
            // bf16 stages of one A and one B plane: one thread runs the issue loop,
            // each stage's MMAs and its commit issued from one block (pairs: from the
            // even CTA, which alone enters with ok set)
            if (lane == 0 && ok) {
                int s = 0;
                uint32_t ph = 0u;  // parity of the full-barrier phase to wait for
                const uint64_t sunits = C::kStage >> 4, bunits = C::kBOff >> 4;
                const uint32_t n16 = static_cast<uint32_t>(p.kin) >> 4;  // MMAs per stage (EPI = 2)
                for (int64_t u = u0; u < n_tiles && ok; u += ustep, ++t) {
                    const int acc = t & 1;
                    // CG = 2: the phase includes arrivals of the odd CTA's epilogue
                    if (t >= 2) ok = tc::mbar_wait<CG == 2>(&S->tmem_empty[acc], ((t / 2) - 1) & 1, abort, p.status);
                    if (!ok) break;
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint32_t d = tmem + static_cast<uint32_t>(acc * kN);
                    for (int ks = 0; ks < nks; ++ks) {
                        // PK pairs: the phase includes the odd CTA's producers (released at cluster scope)
                        ok = tc::mbar_wait<PK && CG == 2>(&S->full[s], ph, abort, p.status);
                        if (!ok) break;
                        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                        const uint64_t ad = bdesc0 + static_cast<uint64_t>(s) * sunits;
                        if constexpr (CG == 2)
                            stage_f16_pair<C::kIdesc>(d, ad, ad + bunits, ks > 0 ? 1u : 0u, empty0 + 8u * s);
                        else
                            if constexpr (EPI == 2)  // short tiles: fewer than four MMAs when R < 64
                                stage_f16<C::kIdesc, MC, true>(d, ad, ad + bunits, ks > 0 ? 1u : 0u, 1u,
                                                               empty0 + 8u * s, n16);
                            else
                                stage_f16<C::kIdesc, MC>(d, ad, ad + bunits, ks > 0 ? 1u : 0u, 1u, empty0 + 8u * s);
                        if (++s == kStages) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                    if (ok) commit(&S->tmem_full[acc]);
                }
            }
            ok = false;  // the generic loop below is not entered
        }
        if constexpr (!TF32 && ASRC == kAHalo) {
            // 3x3 halo tiles, chunk by chunk (halo buffer hb of the ring), the taps in
            // turn: tap (kh, kw) reads the halo from row kh * (Q + 2) + kw on.  One
            // thread runs the issue loop.  Resident weights: the three taps of a
            // kernel row go out as one block of twelve MMAs, and no weight stage is
            // released; otherwise each tap is a stage of the ring.  Descriptors in
            // 16-byte units: + wq_units per halo row of taps, + 8 per column,
            // + hunits per halo buffer, + sunits per stage.
            if (lane == 0 && ok) {
                int hs = 0, hb = 0;
                uint32_t hsph = 0u, hph = 0u;
                const uint64_t wq_units = static_cast<uint64_t>(box.QB + p.KW - 1) * 8u;
                const uint64_t hunits = hbytes >> 4, sunits = C::kStage >> 4;
                const bool res = box.resident != 0;
                for (int64_t u = u0; u < n_tiles && ok; u += ustep, ++t) {
                    const int acc = t & 1;
                    // CG = 2: the phase includes arrivals of the odd CTA's epilogue
                    if (t >= 2) ok = tc::mbar_wait<CG == 2>(&S->tmem_empty[acc], ((t / 2) - 1) & 1, abort, p.status);
                    if (!ok) break;
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint32_t d = tmem + static_cast<uint32_t>(acc * kN);
                    if (res) hs = 0;
                    for (int c = 0; c < hchunks && ok; ++c) {
                        ok = tc::mbar_wait(&S->hfull[hb], hph, abort, p.status);
                        if (!ok) break;
                        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                        const uint64_t hdesc = hdesc0 + static_cast<uint64_t>(hb) * hunits;
                        for (int kh = 0; kh < 3 && ok; ++kh) {
                            const uint64_t arow = hdesc + static_cast<uint64_t>(kh) * wq_units;
                            if (res) {
                                if (t == 0) {  // the row's weights land once, for the first tile
                                    for (int kw = 0; kw < 3 && ok; ++kw)
                                        ok = tc::mbar_wait(&S->full[hs + kw], 0u, abort, p.status);
                                    if (!ok) break;
                                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                                }
                                if constexpr (CG == 1)  // (pairs never keep their weights resident)
                                    row3_f16<C::kIdesc, (C::kStage >> 4)>(
                                        d, arow, bdesc0 + static_cast<uint64_t>(hs) * sunits, (c | kh) != 0 ? 1u : 0u);
                                hs += 3;
                            } else {
                                for (int kw = 0; kw < 3 && ok; ++kw) {
                                    ok = tc::mbar_wait(&S->full[hs], hsph, abort, p.status);
                                    if (!ok) break;
                                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                                    const uint64_t bd = bdesc0 + static_cast<uint64_t>(hs) * sunits;
                                    const uint32_t accf = (c | kh | kw) != 0 ? 1u : 0u;
                                    if constexpr (CG == 2)  // the pair's MMAs; the stage released in both CTAs
                                        stage_f16_pair<C::kIdesc>(d, arow + kw * 8u, bd, accf, empty0 + 8u * hs);
                                    else
                                        stage_f16<C::kIdesc>(d, arow + kw * 8u, bd, accf, 1u, empty0 + 8u * hs);
                                    if (++hs == kStages) {
                                        hs = 0;
                                        hsph ^= 1u;
                                    }
                                }
                            }
                        }
                        if (ok) commit(&S->hempty[hb]);  // CG = 2: the halo buffer freed in both CTAs
                        if (++hb == box.nh) {
                            hb = 0;
                            hph ^= 1u;
                        }
                    }
                    if (ok) commit(&S->tmem_full[acc]);
                }
            }
            ok = false;  // the generic loop below is not entered
        }
        for (int64_t u = u0; u < n_tiles && ok; u += ustep, ++t) {
            const int acc = t & 1;
            // CG = 2: the phase includes arrivals of the odd CTA's epilogue
            if (t >= 2) ok = tc::mbar_wait<CG == 2>(&S->tmem_empty[acc], ((t / 2) - 1) & 1, abort, p.status);
            if (!ok) break;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t d = tmem + static_cast<uint32_t>(acc * kN);
            for (int ks = 0; ks < nks && ok; ++ks, ++it) {
                const int s = it % kStages;
                // PK pairs: the phase includes the odd CTA's producers (released at cluster scope)
                ok = tc::mbar_wait<PK && CG == 2>(&S->full[s], (it / kStages) & 1, abort, p.status);
                if (!ok) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                if (lane == 0) {
                    const uint32_t st = base + s * C::kStage;
                    const uint32_t bst = st + C::kBOff;
                    if constexpr (TF32) {
                        // the split's three terms (stage_tf32_split), A planes in shared memory
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            mma<true, 1>(d, tc::sw128_desc(st + k * 32), tc::sw128_desc(bst + k * 32), C::kIdesc,
                                         (ks > 0 || k > 0) ? 1u : 0u);
#pragma unroll
                        for (int k = 0; k < 2; ++k) {
                            const uint32_t a1 = st + C::kAPlane + k * 32, b1 = bst + C::kBPlane + k * 32;
                            mma<false, 1>(d, tc::sw128_desc(a1), tc::sw128_desc(b1 + 64), C::kIdescB, 1u);
                            mma<false, 1>(d, tc::sw128_desc(a1 + 64), tc::sw128_desc(b1), C::kIdescB, 1u);
                        }
                    } else if constexpr (CG == 2) {
#pragma unroll
                        for (int k = 0; k < kKS / 16; ++k)
                            mma<TF32, CG>(d, tc::sw128_desc(st + k * 32), tc::sw128_desc(bst + k * 32), C::kIdesc,
                                          (ks > 0 || k > 0) ? 1u : 0u);
                    }
                    if constexpr (TF32 || CG == 2) commit(&S->empty[s]);
                }
                if constexpr (!TF32 && CG == 1)
                    stage_f16<C::kIdesc>(d, bdesc0 + static_cast<uint64_t>(s) * (C::kStage >> 4),
                                         bdesc0 + static_cast<uint64_t>(s) * (C::kStage >> 4) + (C::kBOff >> 4),
                                         ks > 0 ? 1u : 0u, issue, empty0 + 8u * s);
                __syncwarp();
            }
            if (ok && lane == 0) commit(&S->tmem_full[acc]);
            __syncwarp();
        }
        if (lane == 0 && (CG == 1 || crank == 0)) commit(&S->drain);
        __syncwarp();
        int no_abort = 0;
        tc::mbar_wait(&S->drain, 0, &no_abort, p.status);
    } else {
        // ------------------------------------------------------------ epilogue (warps 0-3;
        // with EPI = 2 also warps 4-7 as a second group: group g takes the tiles
        // whose accumulator is g)
        constexpr int kEG = C::kEG;
        const int eg = warp >> 2;              // this thread's group
        const int etid = tid - 128 * eg;       // thread within the group; 0 issues its stores
        const int ebar = 1 + eg;               // the group's named barrier
        int t = eg;
        bool ok = true;
        const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
        const int m = etid;  // accumulator row = TMEM lane
        int chunk_no = 0;
        // CG = 2: the odd CTA releases an accumulator on the even CTA's barrier
        const uint32_t tmem_empty_remote = CG == 2 ? map_to_rank(tc::smem_u32(&S->tmem_empty[0]), 0) : 0u;
        for (int64_t u = u0 + eg * ustep; u < n_tiles && ok; u += kEG * ustep, t += kEG) {
            const int acc = t & 1;
            int64_t mt, ct;
            split_unit(u, mt, ct);
            const int co0 = static_cast<int>(ct * kN);
            BoxIdx bi{0, 0, 0};
            if constexpr (ASRC == kA4d || ASRC == kAHalo) bi = box_of(mt, box);
            ok = tc::mbar_wait(&S->tmem_full[acc], (t / 2) & 1, abort, p.status);
            ok = tc::named_and(ebar, 128, ok);
            if (!ok) break;
            __syncwarp();
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const int sc = p.out_bf16 ? 64 : 32;  // output columns per staged 128-byte row
            const int cend = (p.Cout - co0) < kN ? static_cast<int>(p.Cout - co0) : kN;
#pragma unroll 1
            for (int c0 = 0; c0 < cend; c0 += sc, ++chunk_no) {
                uint32_t v[32];
                const uint32_t tcol = tmem + lane_off + static_cast<uint32_t>(acc * kN + c0);
                // output columns of this chunk inside the layer (the store clips the rest):
                // the 16-byte pieces of each staged row that need writing
                const int valid = (cend - c0) < sc ? cend - c0 : sc;
                const int nq = p.out_bf16 ? (valid + 7) / 8 : (valid + 3) / 4;
                if (!p.out_bf16) {
                    tc::tmem_ld32(tcol, v);
                    epilogue_math(v, p, co0 + c0);
                } else {
                    uint32_t w[32];
                    tc::tmem_ld32(tcol, w);
                    epilogue_math(w, p, co0 + c0);
#pragma unroll
                    for (int j = 0; j < 16; ++j) v[j] = bf16x2_rn(w[2 * j], w[2 * j + 1]);
                    if (valid > 32) {  // the second 32 columns (a narrower last chunk has none)
                        tc::tmem_ld32(tcol + 32, w);
                        epilogue_math(w, p, co0 + c0 + 32);
#pragma unroll
                        for (int j = 0; j < 16; ++j) v[16 + j] = bf16x2_rn(w[2 * j], w[2 * j + 1]);
                    }
                }
                if (c0 + sc >= cend) {
                    // the tile's accumulator is all in registers: release it to the MMAs
                    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
                    if (CG == 2 && crank != 0)
                        mbar_arrive_remote(tmem_empty_remote + static_cast<uint32_t>(acc * sizeof(uint64_t)));
                    else
                        tc::mbar_arrive(&S->tmem_empty[acc]);
                }
                // the group's buffers take the chunks in turn; a buffer is rewritten once
                // the store issued from it kYPerGroup chunks earlier has read it
                constexpr int kYG = C::kYPerGroup;
                const uint32_t buf = ybuf + static_cast<uint32_t>(kYG * eg + (chunk_no % kYG)) * C::kYBuf;
                if (etid == 0) tc::bulk_wait_read<kYG - 1>();
                tc::named_sync(ebar, 128);
                // halo tiles: row m = pi * (Q + 2) + qi goes to staged row pi * Q + qi
                // (the box of the store), the two unused columns of each row nowhere
                int srow = m;
                bool stage_row = true;
                if constexpr (ASRC == kAHalo) {
                    const int wq = box.QB + p.KW - 1;
                    const int pi = m / wq, qi = m - (m / wq) * wq;
                    srow = pi * box.QB + qi;
                    stage_row = pi < box.PB && qi < box.QB;
                }
                if (stage_row) {
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        if (q < nq)
                            st_shared_v4(buf + sw_chunk(srow, q), v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                }
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                tc::named_sync(ebar, 128);
                if (etid == 0) {
                    if constexpr (ASRC == kA4d || ASRC == kAHalo)
                        tc::tma_store_4d(&tmY, buf, co0 + c0, bi.qb * box.QB, bi.pb * box.PB,
                                         static_cast<int>(bi.bb * box.BB));
                    else
                        tc::tma_store_2d(&tmY, buf, co0 + c0, static_cast<int>(mt * kM));
                    tc::bulk_commit();
                }
            }
        }
        if (etid == 0) tc::bulk_wait_all();
    }

    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    // CG = 2: neither CTA leaves (or frees tensor memory) while the other may still
    // signal its barriers or the pair's MMAs may read its shared memory
    if constexpr (C::kPairUnits) cluster_sync();
    if (warp == 8) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        if constexpr (CG == 2)
            asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::kTmemCols)
                         : "memory");
        else
            asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::kTmemCols)
                         : "memory");
    }
}

// ---------------------------------------------------------------------------
// host: tensor maps, tile choice and launch
// ---------------------------------------------------------------------------
inline PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess)
            return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
        return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    }();
    return fn;
}

// map over `rank` dims (dims[0] innermost, element counts) with byte strides
// strides[i] of dims 1.., box[] elements per dim, 128-byte swizzle (box[0] * elem
// must be 128) unless `swizzle` is false (box[0] * elem a multiple of 16); false
// if the driver rejects it
inline bool make_map_strided(CUtensorMap *m, const void *ptr, CUtensorMapDataType dt, int rank,
                             const int64_t *dims, const int64_t *strides, const int *box, bool swizzle = true)
{
    auto fn = encode_fn();
    if (!fn || rank < 1 || rank > 5) return false;
    cuuint64_t gd[5], gs[4];
    cuuint32_t bx[5], es[5];
    for (int i = 0; i < rank; ++i) {
        if (dims[i] < 1) return false;
        gd[i] = static_cast<cuuint64_t>(dims[i]);
        bx[i] = static_cast<cuuint32_t>(box[i]);
        es[i] = 1;
        if (i > 0) gs[i - 1] = static_cast<cuuint64_t>(strides[i - 1]);
    }
    return fn(m, dt, static_cast<cuuint32_t>(rank), const_cast<void *>(ptr), gd, gs, bx, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// the same over a packed row-major array
inline bool make_map(CUtensorMap *m, const void *ptr, CUtensorMapDataType dt, int elem, int rank,
                     const int64_t *dims, const int *box)
{
    int64_t strides[4];
    int64_t s = elem;
    for (int i = 0; i + 1 < rank && i < 4; ++i) {
        s *= dims[i];
        strides[i] = s;
    }
    return make_map_strided(m, ptr, dt, rank, dims, strides, box);
}

// activation maps of the layer for source asrc (stage depth ks elements); false
// if a map cannot be encoded
inline bool build_a_maps(const FwdParams &p, const ConvBox &box, int asrc, bool tf32, int ks, AMaps *am)
{
    const CUtensorMapDataType dt = tf32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const int64_t e = tf32 ? 4 : 2;
    if (asrc == kA2d) {
        const int64_t dims[2] = {p.Cin, p.N};
        const int bx[2] = {ks, 128};
        return make_map(&am->m[0], p.X, dt, static_cast<int>(e), 2, dims, bx);
    }
    if (asrc == kAHalo) {
        // the halo of PB output rows: Q + KW - 1 columns by PB + KH - 1 rows of
        // input pixels, 64 channels, from (q, p) = (-pw, p0 - ph) on
        const int64_t dims[4] = {p.Cin, p.W, p.H, box.B};
        const int64_t strides[3] = {p.Cin * e, p.W * p.Cin * e, p.H * p.W * p.Cin * e};
        const int bx[4] = {64, box.QB + p.KW - 1, box.PB + p.KH - 1, 1};
        return make_map_strided(&am->m[0], p.X, dt, 4, dims, strides, bx);
    }
    if (asrc != kA4d) return true;
    for (int rh = 0; rh < p.sh; ++rh)
        for (int rw = 0; rw < p.sw; ++rw) {
            const char *base = static_cast<const char *>(p.X) + (rh * p.W + rw) * p.Cin * e;
            const int64_t dims[4] = {p.Cin, (p.W - rw + p.sw - 1) / p.sw, (p.H - rh + p.sh - 1) / p.sh, box.B};
            const int64_t strides[3] = {p.sw * p.Cin * e, p.sh * p.W * p.Cin * e, p.H * p.W * p.Cin * e};
            const int bx[4] = {ks, box.QB, box.PB, box.BB};
            if (!make_map_strided(&am->m[rh * p.sw + rw], base, dt, 4, dims, strides, bx)) return false;
        }
    return true;
}

inline int sm_count()
{
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return sms > 0 ? sms : 1;
}

// the output-pixel box with the fewest M tiles (ties: longer runs along q, then
// p).  Only the smallest box of each tile count along q and p is tried.
inline ConvBox choose_box(int64_t B, int64_t P, int64_t Q)
{
    ConvBox best{1, 1, 1, 1, 1, 1, B};
    int64_t best_tiles = -1;
    for (int64_t QB = 1; QB <= Q && QB <= 128; ++QB) {
        const int64_t nq = (Q + QB - 1) / QB;
        if ((Q + nq - 1) / nq != QB) continue;
        for (int64_t PB = 1; PB <= P && QB * PB <= 128; ++PB) {
            const int64_t np = (P + PB - 1) / PB;
            if ((P + np - 1) / np != PB) continue;
            const int64_t BB = (128 / (QB * PB)) < B ? 128 / (QB * PB) : B;
            const int64_t tiles = nq * np * ((B + BB - 1) / BB);
            if (best_tiles < 0 || tiles <= best_tiles) {
                best_tiles = tiles;
                best.QB = static_cast<int>(QB);
                best.PB = static_cast<int>(PB);
                best.BB = static_cast<int>(BB);
            }
        }
    }
    best.nQ = static_cast<int>((Q + best.QB - 1) / best.QB);
    best.nP = static_cast<int>((P + best.PB - 1) / best.PB);
    best.rows = best.QB * best.PB * best.BB;
    best.B = B;
    return best;
}

// the activation source of a layer for stage depth ks (elements per 128-byte row)
inline int a_source(const FwdParams &p, int ks)
{
    const int64_t lim = int64_t(1) << 30;
    if (!p.is_conv) return p.N < lim ? kA2d : kAGather;
    const bool fits = p.H < lim && p.W < lim && p.N < lim && (p.N / (p.P * p.Q)) < lim;
    const bool strides_ok = p.sh >= 1 && p.sh <= 2 && p.sw >= 1 && p.sw <= 2 && p.H >= p.sh && p.W >= p.sw;
    return (strides_ok && p.Cin % ks == 0 && fits) ? kA4d : kAGather;
}

// N tile among {64, 128, 256} (up to max_bn): fewest rounds of tiles over the
// SMs (CG = 2: pair tiles over the SM pairs) weighted by the tile's width plus a
// fixed per-tile cost; ties: the wider
inline int choose_bn(int64_t m_tiles, int64_t Cout, int max_bn, int cg = 1)
{
    const int64_t sms = sm_count() / cg;
    int best = 64;
    int64_t best_cost = -1;
    for (int bn = 64; bn <= max_bn; bn *= 2) {
        const int64_t tiles = ((m_tiles + cg - 1) / cg) * ((Cout + bn - 1) / bn);
        const int64_t cost = ((tiles + sms - 1) / sms) * (bn + 32);
        if (best_cost < 0 || cost <= best_cost) {
            best_cost = cost;
            best = bn;
        }
    }
    return best;
}

// reduction indices a stage copies: the stage depth, or for bf16 products with
// fewer than 64 indices (one stage) the indices rounded up to 16: narrower copies
// (no out-of-range fill for three quarters of the box when R = 16) and one MMA per
// 16 indices (measured on the MobileNetV2 pointwise layers of 16-32 input channels:
// 20-35 % faster)
inline int stage_k_in(const FwdParams &p, bool tf32, int asrc, bool pk)
{
    if (tf32) return 32;
    if (pk || asrc != kA2d || p.R >= 64) return 64;
    return static_cast<int>((p.R + 15) / 16 * 16);
}

template <bool TF32, int ASRC, int BN, int CG, int EPI = 1, bool PK = false, bool MC = false>
cudaError_t launch_cfg(const FwdParams &p, const ConvBox &box_in, const AMaps &tmA, cudaStream_t stream)
{
    using C = Cfg<TF32, ASRC, BN, CG, EPI, PK, MC>;
    auto kern = gemm_ws_kernel<TF32, ASRC, BN, CG, EPI, PK, MC>;
    ConvBox box = box_in;
    size_t smem = C::kSmem;
    if constexpr (C::kHalo) {
        // the halo ring takes the shared memory left: up to kMaxHalo buffers, two at least
        const size_t hb = static_cast<size_t>(box.hrows) * 128;
        const size_t left = kMaxSmemPerBlock - C::kSmem;
        box.nh = static_cast<int>(left / hb < static_cast<size_t>(tc::kMaxHalo) ? left / hb : tc::kMaxHalo);
        if (box.nh < 2) return cudaErrorInvalidValue;
        smem += static_cast<size_t>(box.nh) * hb;
    }
    static SmemAttrCache attr_cache;
    const cudaError_t attr = smem_attr_once(
        kern, static_cast<int>(C::kHalo ? static_cast<size_t>(kMaxSmemPerBlock) : C::kSmem), attr_cache);
    if (attr != cudaSuccess) return attr;
    CUtensorMap tmB0{}, tmB1{}, tmY{};
    const CUtensorMapDataType dt = TF32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    const int elem = TF32 ? 4 : 2;
    const int64_t wdims[2] = {p.R, p.Cout};
    FwdParams q = p;
    // narrower stage copies only in the short-tile form (one-stage layers land there)
    q.kin = EPI == 2 ? stage_k_in(p, TF32, ASRC, PK) : C::kKS;
    const int wbox[2] = {q.kin, MC ? C::kBRows / 2 : C::kBRows};  // MC: each CTA copies half the rows
    if (!PK && !make_map(&tmB0, p.wdense, dt, elem, 2, wdims, wbox)) return cudaErrorInvalidValue;
    if (!PK && C::kBPlanes > 1) {
        // fp32: plane 1 of the split, bf16 [Cout][ceil(R / 32) * 64], one 128-byte row per stage
        const char *pl1 = static_cast<const char *>(p.wdense) + static_cast<size_t>(p.Cout) * p.R * elem;
        const int64_t dims1[2] = {(p.R + 31) / 32 * 64, p.Cout};
        const int box1[2] = {64, MC ? C::kBRows / 2 : C::kBRows};
        if (!make_map(&tmB1, pl1, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, 2, dims1, box1)) return cudaErrorInvalidValue;
    }
    // output rows of 128 bytes: 32 fp32 or 64 bf16 channels
    const CUtensorMapDataType ydt = p.out_bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    const int yel = p.out_bf16 ? 2 : 4, ysc = p.out_bf16 ? 64 : 32;
    if constexpr (ASRC == kA4d || ASRC == kAHalo) {
        const int64_t dims[4] = {p.Cout, p.Q, p.P, box.B};
        const int bx[4] = {ysc, box.QB, box.PB, box.BB};
        if (!make_map(&tmY, p.Y, ydt, yel, 4, dims, bx)) return cudaErrorInvalidValue;
    } else {
        const int64_t dims[2] = {p.Cout, p.N};
        const int bx[2] = {ysc, C::kM};
        if (!make_map(&tmY, p.Y, ydt, yel, 2, dims, bx)) return cudaErrorInvalidValue;
    }
    const int64_t n_ct = (p.Cout + C::kN - 1) / C::kN;
    if constexpr (C::kHalo && !PK && CG == 1)  // resident weights: single-CTA tiles
        box.resident = (n_ct == 1 && (p.R + C::kKS - 1) / C::kKS <= C::kStages) ? 1 : 0;
    const int64_t m_tiles = (ASRC == kA4d || ASRC == kAHalo)
                                ? static_cast<int64_t>(box.nQ) * box.nP * ((box.B + box.BB - 1) / box.BB)
                                         : (p.N + C::kM - 1) / C::kM;
    // CG = 2 or MC: units are pair tiles (two M tiles), one per cluster of two CTAs
    constexpr int kCl = C::kPairUnits ? 2 : 1;
    const int64_t n_tiles = n_ct * (kCl == 2 ? (m_tiles + 1) / 2 : m_tiles);
    const int64_t slots = sm_count() / kCl;
    const int64_t grid = kCl * (n_tiles < slots ? n_tiles : slots);
    // programmatic dependent launch: may start once every block of the preceding
    // kernel on the stream (the decompression) has signalled; it waits for that
    // kernel's completion before reading memory
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(C::kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute la[2];
    la[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    la[0].val.programmaticStreamSerializationAllowed = 1;
    la[1].id = cudaLaunchAttributeClusterDimension;
    la[1].val.clusterDim.x = kCl;
    la[1].val.clusterDim.y = 1;
    la[1].val.clusterDim.z = 1;
    cfg.attrs = la;
    cfg.numAttrs = kCl == 2 ? 2 : 1;
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, q, tmA, tmB0, tmB1, tmY, box, n_ct, n_tiles);
    return e != cudaSuccess ? e : cudaGetLastError();
}

// activation source, pixel box and activation maps of a layer (stage depth ks):
// the 4-D copy when the layer allows it and its maps encode, else the gather
struct Plan {
    int asrc;
    ConvBox box;
    AMaps am;
};
// halo box of a bf16 3x3, stride-1, padding-1 convolution: PB output rows of
// the full width per tile.  Used for layers of 256 input channels or more (four
// chunks or more per tile: the per-tap copies there move 9 x the halo's bytes,
// and the halo copies measured 7-11 % faster on the 14 x 14 ResNet-50 layers;
// with 64 or 128 channels the tile is bound by the MMAs' shared-memory reads
// and the per-tap form measured faster), and for 64 -> 64 layers, whose nine
// weight tiles stay resident in the stages (no per-tap weight copies either),
// whose output rows per tile are at least three quarters of the 4-D box's
// (images narrower than the tile fit several per 4-D box, not per halo)
inline bool halo_box(const FwdParams &p, const ConvBox &a4d, ConvBox *hb)
{
    if (!(p.is_conv && p.KH == 3 && p.KW == 3 && p.sh == 1 && p.sw == 1 && p.ph == 1 && p.pw == 1 &&
          p.Cin % 64 == 0 && (p.Cin >= 256 || (p.Cin == 64 && p.Cout <= 64)) && p.P == p.H && p.Q == p.W &&
          p.Q + 2 <= 66))
        return false;
    const int wq = static_cast<int>(p.Q) + 2;
    const int pb = static_cast<int>(p.P < 128 / wq ? p.P : 128 / wq);
    if (pb < 1 || 4 * pb * p.Q < 3 * a4d.rows) return false;
    const int64_t B = p.N / (p.P * p.Q);
    // rows an MMA can read: 128 from the largest tap offset 2 * wq + 2 on, in
    // whole 1024-byte swizzle patterns
    const int hrows = (128 + 2 * wq + 2 + 7) / 8 * 8;
    *hb = ConvBox{static_cast<int>(p.Q), pb, 1, 1, static_cast<int>((p.P + pb - 1) / pb), pb * wq, B, hrows, 0};
    return true;
}

inline void plan_layer(const FwdParams &p, bool tf32, int ks, Plan *pl)
{
    pl->asrc = a_source(p, ks);
    pl->box = ConvBox{1, 1, 1, 1, 1, 1, 1};
    if (pl->asrc == kA4d) pl->box = choose_box(p.N / (p.P * p.Q), p.P, p.Q);
    ConvBox hb;
    if (pl->asrc == kA4d && !tf32 && halo_box(p, pl->box, &hb)) {
        pl->asrc = kAHalo;
        pl->box = hb;
    }
    if (!build_a_maps(p, pl->box, pl->asrc, tf32, ks, &pl->am)) {
        pl->asrc = kAGather;
        pl->box = ConvBox{1, 1, 1, 1, 1, 1, 1};
    }
}

// m tiles of the layer for the chosen activation source
inline int64_t m_tiles_of(const FwdParams &p, int asrc, const ConvBox &box)
{
    if (asrc == kA4d || asrc == kAHalo)
        return static_cast<int64_t>(box.nQ) * box.nP * ((box.B + box.BB - 1) / box.BB);
    return (p.N + 127) / 128;
}

}  // namespace ws
}  // namespace cci
