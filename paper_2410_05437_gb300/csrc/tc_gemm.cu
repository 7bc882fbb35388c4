// tc_gemm.cu -- persistent, warp-specialized tcgen05 GEMM for sm_103a.
//
// One CTA per SM loops over output tiles of 128 x BN. Warp 0 (one lane) streams A and B
// tiles into a STAGES-deep shared-memory ring with TMA (128-byte swizzle); warp 1 (one lane)
// issues tcgen05.mma (bf16 x bf16 -> fp32) into one of two TMEM accumulators; warps 2-5
// drain the other accumulator with tcgen05.ld and write the tile, so the epilogue of tile i
// overlaps the main loop of tile i+1. mbarriers link the roles; every wait is bounded.
//
// Two operand layouts share the kernel:
//   * K-major ("TN"): C[r][c] = sum_k A[r][k] B[c][k] -- the projected layer's two products
//     Z = X P and Y = Z W' (with P^T and W'^T stored row-major), the fold W'^T = W P and
//     the dense baseline Y = X W^T. For few tokens the operands swap (A = the weights, 128
//     rows per tile; B = the tokens) and the epilogue stores the tile transposed, so that
//     the grid spans the weight rows; a reduction split over CTAs writes fp32 partial tiles
//     to a workspace, and a second launch adds them in split order (deterministic) and
//     stores the bf16 result;
//   * M/N-major: S[i][j] += sum_t X[t][i] X[t][j] -- the autocorrelation of Eq. 4, read
//     straight from token-major X, upper-triangle tiles only, split over tokens with fp32
//     atomics.
#include <cuda.h>
#include <cuda_runtime.h>

#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <vector>

#include "../../include/espace.h"
#include "kernels.h"
#include "ptx.cuh"

namespace espace {

constexpr int BM = 128;                 // UMMA M: rows per tile (= TMEM lanes)
constexpr int BK = 64;                  // bf16 elements per 128-byte swizzled row
constexpr int UMMA_K = 16;              // K of one tcgen05.mma.kind::f16
constexpr int EPI_THREADS = 128;        // 4 epilogue warps, one per TMEM lane quarter
constexpr int GEMM_THREADS = 64 + EPI_THREADS;

enum { EPI_STORE_BF16 = 0, EPI_ATOMIC_UPPER_F32 = 1, EPI_STORE_BF16_T = 2, EPI_SPLIT_BF16_T = 3 };

struct TcGemmArgs {
    int rows, cols;        // output extent
    int kblocks;           // 64-wide blocks along the reduction
    int tiles_n;           // column tiles (row-major tile grid when tile_list == nullptr)
    int num_tiles;         // output tiles
    int ksplit;            // reduction splits per tile (EPI_ATOMIC_UPPER_F32, EPI_SPLIT_BF16_T)
    int kb_per_split;
    const int2* tile_list; // (tile row, tile col) pairs, or nullptr
    void* out;
    int64_t ldo;
    // EPI_SPLIT_BF16_T: fp32 partial of split s, row r at part[(s * rows + r) * ld_part]
    float* part;
    int64_t ld_part;
    // K-major only: rows of each B tile load (0: BN). Fewer than BN when B has fewer rows:
    // the tile's other rows keep stale shared memory, which reaches only output columns past
    // `cols` (never stored) -- cheaper than the copy engine's zero fill of absent rows
    int b_rows;
    // K-major only, launched with programmatic stream serialization: A (weights the caller
    // guarantees the preceding grid does not write) is loaded for the first STAGES k-blocks
    // before waiting for the preceding grid; B (tokens, maybe its output) only after
    int pdl;
    int* status;
    uint64_t wait_limit_ns;
};

template <int BN, int STAGES>
struct TcCfg {
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int TMEM_COLS = 2 * BN;
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + 256;
    static_assert(STAGE_BYTES % 1024 == 0, "stages must keep 1024-byte alignment");
    static_assert(TMEM_COLS <= 512, "two accumulators must fit in TMEM");
};

// After a producer gave up, copies it already issued may still be landing in shared
// memory: wait 200 us (far longer than any copy takes) before the CTA can exit.
__device__ __forceinline__ void settle_copies()
{
    const uint64_t t0 = globaltimer_ns();
    while (globaltimer_ns() - t0 < 200000ull) __nanosleep(1000);
}

__device__ __forceinline__ void decode_item(const TcGemmArgs& a, int item, int& tm, int& tn,
                                            int& kb0, int& kb1)
{
    const int tile = item / a.ksplit;
    const int split = item - tile * a.ksplit;
    if (a.tile_list != nullptr) {
        const int2 t = a.tile_list[tile];
        tm = t.x;
        tn = t.y;
    } else {
        tm = tile / a.tiles_n;
        tn = tile - tm * a.tiles_n;
    }
    kb0 = split * a.kb_per_split;
    kb1 = min(kb0 + a.kb_per_split, a.kblocks);
}

template <int BN, int STAGES, bool MN_MAJOR, int EPI>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap map_a,
                   const __grid_constant__ CUtensorMap map_b, const TcGemmArgs args)
{
    using Cfg = TcCfg<BN, STAGES>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * Cfg::STAGE_BYTES);
    uint64_t* empty = full + STAGES;
    uint64_t* tfull = empty + STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], EPI_THREADS);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    if (warp == 0 && lane == 0) {
        tma_prefetch_map(&map_a);
        tma_prefetch_map(&map_b);
    }
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;

    const int num_items = args.num_tiles * args.ksplit;
    const uint64_t limit = args.wait_limit_ns;

    if (args.pdl && threadIdx.x == 0) grid_dep_launch_dependents();

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            // B loads held back until the preceding grid has completed (pdl)
            bool dep_done = MN_MAJOR || !args.pdl;
            int ndef = 0;
            int def_stage[STAGES], def_kb[STAGES], def_tn[STAGES];
            auto release_deferred = [&]() {
                grid_dep_wait();
                for (int q = 0; q < ndef; ++q)
                    tma_load_2d(smem + def_stage[q] * Cfg::STAGE_BYTES + Cfg::A_BYTES, &map_b, &full[def_stage[q]],
                                def_kb[q] * BK, def_tn[q] * BN);
                ndef = 0;
                dep_done = true;
            };
            for (int item = blockIdx.x; ok && item < num_items; item += gridDim.x) {
                int tm, tn, kb0, kb1;
                decode_item(args, item, tm, tn, kb0, kb1);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!dep_done && ndef == STAGES) release_deferred();
                    if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, args.status, limit,
                                   ESPACE_ERR_TIMEOUT)) {
                        ok = false;
                        break;
                    }
                    uint8_t* sa = smem + stage * Cfg::STAGE_BYTES;
                    uint8_t* sb = sa + Cfg::A_BYTES;
                    mbar_arrive_expect_tx(&full[stage], (!MN_MAJOR && args.b_rows > 0)
                                                            ? static_cast<uint32_t>(Cfg::A_BYTES + args.b_rows * BK * 2)
                                                            : static_cast<uint32_t>(Cfg::STAGE_BYTES));
                    if (MN_MAJOR) {
                        // 64 features x 64 tokens per box; box h of a tile at +h*8 KB
                        tma_load_2d(sa, &map_a, &full[stage], tm * BM, kb * BK);
                        tma_load_2d(sa + 8192, &map_a, &full[stage], tm * BM + 64, kb * BK);
#pragma unroll
                        for (int h = 0; h < BN / 64; ++h)
                            tma_load_2d(sb + h * 8192, &map_b, &full[stage], tn * BN + h * 64,
                                        kb * BK);
                    } else {
                        tma_load_2d(sa, &map_a, &full[stage], kb * BK, tm * BM);
                        if (dep_done) {
                            tma_load_2d(sb, &map_b, &full[stage], kb * BK, tn * BN);
                        } else {
                            def_stage[ndef] = stage;
                            def_kb[ndef] = kb;
                            def_tn[ndef] = tn;
                            ++ndef;
                        }
                    }
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!dep_done) release_deferred();   // also after giving up: the stages expect B
            if (!ok) settle_copies();
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, MN_MAJOR, MN_MAJOR);
            // K-major: the next 16-element K slice starts 32 bytes further along the
            // swizzled row. MN-major: 16 tokens further = 16 rows of 128 bytes.
            constexpr uint32_t k_step = MN_MAJOR ? 2048u : 32u;
            constexpr uint32_t lbo = MN_MAJOR ? 8192u : 16u;
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int item = blockIdx.x; ok && item < num_items; item += gridDim.x) {
                int tm, tn, kb0, kb1;
                decode_item(args, item, tm, tn, kb0, kb1);
                if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, args.status, limit,
                               ESPACE_ERR_TIMEOUT))
                    break;
                tc_fence_after_sync();
                const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait(&full[stage], phase, abort_flag, args.status, limit,
                                   ESPACE_ERR_TIMEOUT)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t a_addr = smem_u32(smem + stage * Cfg::STAGE_BYTES);
                    const uint32_t b_addr = a_addr + Cfg::A_BYTES;
#pragma unroll
                    for (int j = 0; j < BK / UMMA_K; ++j) {
                        const uint64_t ad = smem_desc_sw128(a_addr + j * k_step, lbo, 1024);
                        const uint64_t bd = smem_desc_sw128(b_addr + j * k_step, lbo, 1024);
                        umma_bf16(d_tmem, ad, bd, idesc, (kb > kb0 || j > 0) ? 1u : 0u);
                    }
                    umma_commit(&empty[stage]);   // frees the stage once these MMAs finish
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                umma_commit(&tfull[acc]);          // accumulator ready for the epilogue
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1u;
            }
            // every MMA issued above has finished once this commit arrives
            umma_commit(drain);
            volatile int never = 0;
            mbar_wait(drain, 0, &never, args.status, cleanup_limit(limit), ESPACE_ERR_TIMEOUT);
        }
    } else {
        // ------------------------------------------------------------ epilogue (4 warps)
        const int quarter = warp & 3;            // TMEM lanes this warp may read
        const int row_in_tile = quarter * 32 + lane;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int item = blockIdx.x; item < num_items; item += gridDim.x) {
            int tm, tn, kb0, kb1;
            decode_item(args, item, tm, tn, kb0, kb1);
            if (!mbar_wait(&tfull[acc], acc_phase, abort_flag, args.status, limit,
                           ESPACE_ERR_TIMEOUT))
                break;
            tc_fence_after_sync();
            const int row = tm * BM + row_in_tile;
            const uint32_t t_row =
                tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(acc * BN);
#pragma unroll 1
            for (int c = 0; c < BN; c += 32) {
                const int col0 = tn * BN + c;
                if (col0 >= args.cols) break;    // uniform across the warp
                uint32_t v[32];
                tmem_ld_32cols(t_row + static_cast<uint32_t>(c), v);
                tmem_ld_wait();
                if (row >= args.rows) continue;
                if (EPI == EPI_STORE_BF16) {
                    __nv_bfloat16* out_row =
                        reinterpret_cast<__nv_bfloat16*>(args.out) + static_cast<int64_t>(row) * args.ldo;
                    if (col0 + 32 <= args.cols) {
                        uint4* dst = reinterpret_cast<uint4*>(out_row + col0);
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            uint4 q;
                            q.x = pack_bf16x2(__uint_as_float(v[8 * i + 0]), __uint_as_float(v[8 * i + 1]));
                            q.y = pack_bf16x2(__uint_as_float(v[8 * i + 2]), __uint_as_float(v[8 * i + 3]));
                            q.z = pack_bf16x2(__uint_as_float(v[8 * i + 4]), __uint_as_float(v[8 * i + 5]));
                            q.w = pack_bf16x2(__uint_as_float(v[8 * i + 6]), __uint_as_float(v[8 * i + 7]));
                            dst[i] = q;
                        }
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (col0 + i < args.cols)
                                out_row[col0 + i] = __float2bfloat16_rn(__uint_as_float(v[i]));
                    }
                } else if (EPI == EPI_ATOMIC_UPPER_F32) {
                    float* out_row =
                        reinterpret_cast<float*>(args.out) + static_cast<int64_t>(row) * args.ldo;
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const int col = col0 + i;
                        if (col < args.cols && col >= row) atomicAdd(out_row + col, __uint_as_float(v[i]));
                    }
                } else if (EPI == EPI_STORE_BF16_T) {
                    // out[col][row]: the warp's 32 lanes hold 32 consecutive rows
                    __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(args.out) + row;
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (col0 + i < args.cols)
                            o[static_cast<int64_t>(col0 + i) * args.ldo] = __float2bfloat16_rn(__uint_as_float(v[i]));
                } else {
                    // this split's fp32 partial (columns up to the next multiple of 32)
                    const int split = item - (item / args.ksplit) * args.ksplit;
                    float4* dst = reinterpret_cast<float4*>(
                        args.part + (static_cast<int64_t>(split) * args.rows + row) * args.ld_part + col0);
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        dst[i] = make_float4(__uint_as_float(v[4 * i]), __uint_as_float(v[4 * i + 1]),
                                             __uint_as_float(v[4 * i + 2]), __uint_as_float(v[4 * i + 3]));
                }
            }
            tc_fence_before_sync();
            mbar_arrive(&tempty[acc]);
            acc ^= 1;
            if (acc == 0) acc_phase ^= 1u;
        }
    }

    __syncwarp();
    tc_fence_before_sync();
    // a role that gave up may leave copies in flight into shared memory: let them land
    if (threadIdx.x == 0 && *abort_flag) settle_copies();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem_base, Cfg::TMEM_COLS);
    }
}

// =========================================================================== CTA-pair kernel
//
// Same pipeline on a pair of CTAs (a cluster of two on neighbouring SMs) computing
// 256 x 256 output tiles with tcgen05.mma.cta_group::2: each CTA stages 128 rows of A and
// 128 rows (half) of B per k-block, so each SM moves 32 KB instead of 48 KB of operands per
// 64-deep k-block for twice the tile. The leader CTA (rank 0) issues the MMAs for both; the
// two producers count their copies on the leader's "full" barrier; the leader's commits
// arrive on both CTAs' "empty" and "accumulator full" barriers; each CTA drains its own
// TMEM half (rows rank*128 .. +128 of the tile) and releases the accumulator on the
// leader's barrier.
constexpr int PAIR_BM = 256;        // tile rows per pair (128 per CTA)
constexpr int PAIR_BN = 256;        // tile columns per pair (B rows: 128 per CTA)
constexpr int PAIR_STAGES = 6;
constexpr int PAIR_A_BYTES = 128 * BK * 2;
constexpr int PAIR_B_BYTES = 128 * BK * 2;
constexpr int PAIR_STAGE_BYTES = PAIR_A_BYTES + PAIR_B_BYTES;
constexpr int PAIR_ACCS = 2;        // TMEM accumulators per CTA (1 or 2)
constexpr int PAIR_TMEM_COLS = PAIR_ACCS * PAIR_BN;
// Work items in flight between the leader's producer and the other roles (see PairArgs).
constexpr int PAIR_RING = 16;
// bf16 epilogue: each warp stages a 32-row x 64-column slice of its tile (4 KB, the
// 128-byte swizzle of the output tensor map) in one of two buffers and stores it with TMA
constexpr int PAIR_EPI_BUF = 32 * 128;
constexpr int PAIR_EPI_BYTES = 4 * 2 * PAIR_EPI_BUF;
// The autocorrelation restarts its TMEM accumulator every SYRK_CHUNK k-blocks (1024
// tokens) and its epilogue adds the chunks in fp32 registers, so that long token runs do
// not lose precision in the tensor core's accumulator.
constexpr int SYRK_CHUNK = 16;
// Longest wait of a pair for the previous wave of items (PairArgs::wave_ctr).
constexpr uint64_t WAVE_WAIT_NS = 20000;
// Tile rows per group of the grouped tile order of full-grid products.
constexpr int PAIR_GROUP_M = 8;
// Diagonal blocks of a block-diagonal product (one per tensor-parallel rank).
constexpr int PAIR_MAX_BLOCKS = 8;
constexpr int PAIR_MAX_SEGS = 6;

template <bool SYRK>
struct PairShape {
    static constexpr int EPI_WARPS = SYRK ? 8 : 4;   // SYRK: two warps per TMEM lane quarter
    static constexpr int THREADS = 64 + 32 * EPI_WARPS;
    static constexpr int STAGING = SYRK ? 0 : PAIR_EPI_BYTES;   // epilogue staging (bf16 stores)
    static constexpr int SMEM_BYTES = 1024 + PAIR_STAGES * PAIR_STAGE_BYTES + STAGING + 512;
    static_assert(SMEM_BYTES <= 232448, "shared memory per CTA");
};

// One product C[rows][cols] = A[rows][k] B[cols][k]^T of a pair program.
struct PairProblem {
    int rows, cols, kblocks, tiles_n;
    int num_tiles;           // output tiles
    int ksplit;              // reduction splits per tile (work items = num_tiles * ksplit)
    int kb_per_split;
    const int2* tile_list;   // (tile row, tile col) pairs, or nullptr for the full grid
    void* out;
    int64_t ldo;
    // token-reduction (M/N-major) programs: bit 0 = add only column >= row; bit 1 (with
    // ksplit == 1 only) = store the tile instead of adding it
    int upper;
    // bf16 programs: 1 = store through the output tensor map (TMA), 0 = direct stores
    int tma_store;
};

// A program of one product, or of two where the second one's A operand is the first one's
// output (the projected layer: Z = X P, then Y = Z W'). Row block tm of the second
// product's A is read only after both CTAs of every tile in row block tm of the first
// product have stored it: ready[tm] counts the epilogue warps that stored their rows
// (target 8 x tiles_n of product 0: four warps in each of two CTAs per tile).
//
// Work items: the leader CTA's producer draws them and hands each to every role of both
// CTAs through a ring in shared memory. With a ticket counter (the two-product program)
// the items are drawn from it with atomics, so they start in one global order, first
// product first, and only pairs that are running draw any: a pair that draws a tile of
// the second product knows that every tile of the first was drawn by a running pair, so
// its wait ends even when some CTA pairs of the grid are not resident (SMs held by other
// work). Without a ticket a pair takes items pair, pair + npairs, ... The last CTA to
// leave (exit counter) zeroes ready[0 .. nready), the ticket and the exit counter, on
// every exit path, so the next launch starts from zero even after one that gave up.
//
// Block-diagonal product (problem 0 of a one-product program, nblocks > 0): output column
// block g, columns [c0[g], c0[g] + cw[g]), is A[:, ak0[g] .. ak0[g] + kdim) times rows
// [c0[g], c0[g] + cw[g]) of B [total cols][kdim] transposed; its column tiles are
// tile0[g] .. tile0[g + 1] - 1 of the tile grid. kdim is a multiple of the 64-deep k-block,
// so a block never reads another block's A columns; B rows of a tile past its block's end
// belong to the next block and only feed columns that are not stored.
struct PairArgs {
    PairProblem p[2];
    int nprob;
    int* ready;
    int nready;
    int* ticket;      // work-item ticket, or nullptr for the static order
    int* exit_ctr;    // CTAs that left (with a ticket or a wave counter)
    // token-reduction programs over many waves of items (static order): items whose loads
    // both CTAs of their pair have issued. A pair starts its i-th item once every pair has
    // issued the loads of its (i-1)-th, so that the pairs of a wave stream the same token
    // rows of the feature slices they share, and those rows are read from L2; the wait is
    // only a hint (at most WAVE_WAIT_NS), and nothing depends on it for correctness
    int* wave_ctr;
    int* status;
    uint64_t wait_limit_ns;
    int nblocks;
    int tile0[PAIR_MAX_BLOCKS + 1];
    int ak0[PAIR_MAX_BLOCKS];
    int c0[PAIR_MAX_BLOCKS];
    int cw[PAIR_MAX_BLOCKS];
    // token-reduction programs: when seg_n > 0, k-block kb is 64-row slab kb / seg_n of
    // segment kb % seg_n, whose A rows start at seg_a[kb % seg_n] and B rows at seg_b[..]:
    // the segments' products over one slab run back to back, so that the operand slabs they
    // share are read from L2
    int seg_n;
    int seg_a[PAIR_MAX_SEGS];
    int seg_b[PAIR_MAX_SEGS];
};

// First token row of k-block kb in A's and in B's map (segmented token reductions).
__device__ __forceinline__ void pair_seg_rows(const PairArgs& a, int kb, int& ya, int& yb)
{
    if (a.seg_n <= 0) {
        ya = yb = kb * BK;
        return;
    }
    const int slab = kb / a.seg_n;
    const int seg = kb - slab * a.seg_n;
    const int off = slab * BK;
    int sa = 0, sb = 0;
#pragma unroll
    for (int q = 0; q < PAIR_MAX_SEGS; ++q)
        if (q == seg) {
            sa = a.seg_a[q];
            sb = a.seg_b[q];
        }
    ya = sa + off;
    yb = sb + off;
}

// Column tile tn of problem prob -> A's k offset, B's first row, the first output column
// and the end of the output columns that tile may store. Unrolled selects keep the block
// table out of local memory.
__device__ __forceinline__ void pair_block_of(const PairArgs& a, int prob, int tn, int cols, int& ak0,
                                              int& brow, int& ccol, int& cend)
{
    if (prob != 0 || a.nblocks == 0) {
        ak0 = 0;
        brow = tn * PAIR_BN;
        ccol = tn * PAIR_BN;
        cend = cols;
        return;
    }
    int g = 0;
#pragma unroll
    for (int i = 1; i < PAIR_MAX_BLOCKS; ++i)
        if (i < a.nblocks && tn >= a.tile0[i]) g = i;
    int t0 = 0, k0 = 0, c0 = 0, cw = 0;
#pragma unroll
    for (int i = 0; i < PAIR_MAX_BLOCKS; ++i)
        if (i == g) {
            t0 = a.tile0[i];
            k0 = a.ak0[i];
            c0 = a.c0[i];
            cw = a.cw[i];
        }
    ak0 = k0;
    brow = c0 + (tn - t0) * PAIR_BN;
    ccol = brow;
    cend = c0 + cw;
}

// Field-wise selection keeps the problem in registers (a dynamic index into the kernel
// parameters would go through local memory).
__device__ __forceinline__ PairProblem pair_problem_of(const PairArgs& a, int prob)
{
    PairProblem r;
    r.rows = prob == 0 ? a.p[0].rows : a.p[1].rows;
    r.cols = prob == 0 ? a.p[0].cols : a.p[1].cols;
    r.kblocks = prob == 0 ? a.p[0].kblocks : a.p[1].kblocks;
    r.tiles_n = prob == 0 ? a.p[0].tiles_n : a.p[1].tiles_n;
    r.num_tiles = prob == 0 ? a.p[0].num_tiles : a.p[1].num_tiles;
    r.ksplit = prob == 0 ? a.p[0].ksplit : a.p[1].ksplit;
    r.kb_per_split = prob == 0 ? a.p[0].kb_per_split : a.p[1].kb_per_split;
    r.tile_list = prob == 0 ? a.p[0].tile_list : a.p[1].tile_list;
    r.out = prob == 0 ? a.p[0].out : a.p[1].out;
    r.ldo = prob == 0 ? a.p[0].ldo : a.p[1].ldo;
    r.upper = prob == 0 ? a.p[0].upper : a.p[1].upper;
    r.tma_store = prob == 0 ? a.p[0].tma_store : a.p[1].tma_store;
    return r;
}

__device__ __forceinline__ int pair_items(const PairProblem& p) { return p.num_tiles * p.ksplit; }

// Work item -> (problem, tile row, tile column, k-block range).
__device__ __forceinline__ void pair_decode(const PairArgs& a, int item, int& prob, int& tm, int& tn,
                                            int& kb0, int& kb1)
{
    const int n0 = a.p[0].num_tiles * a.p[0].ksplit;
    prob = item < n0 ? 0 : 1;
    const PairProblem p = pair_problem_of(a, prob);
    const int j = prob == 0 ? item : item - n0;
    // split-major: consecutive items are consecutive tiles over the same token range, so a
    // wave shares that operand slab in L2 and the splits of one tile, which add into the
    // same output, run at different times
    const int split = j / p.num_tiles, tile = j - split * p.num_tiles;
    if (p.tile_list != nullptr) {
        const int2 t = p.tile_list[tile];
        tm = t.x;
        tn = t.y;
    } else {
        // grouped order: PAIR_GROUP_M tile rows at a time, columns outer within the group, so
        // that the tiles one wave of CTA pairs runs together share A and B slices in L2
        const int tiles_m = p.num_tiles / p.tiles_n;
        const int per_group = PAIR_GROUP_M * p.tiles_n;
        const int first_m = (tile / per_group) * PAIR_GROUP_M;
        const int group_m = min(tiles_m - first_m, PAIR_GROUP_M);
        const int in_group = tile - (tile / per_group) * per_group;
        tm = first_m + in_group % group_m;
        tn = in_group / group_m;
    }
    kb0 = split * p.kb_per_split;
    kb1 = min(kb0 + p.kb_per_split, p.kblocks);
}

__device__ __forceinline__ int ld_acquire_gpu(const int* p)
{
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void red_release_gpu_add(int* p, int v)
{
    asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void fence_proxy_async_global()
{
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

// SYRK = false: K-major A, bf16 stores (the products of Eq. 3 and Eq. 1); B K-major, or with
// B_MN M/N-major (B stored [k][cols], e.g. the weights of a backward product dY W).
// SYRK = true: both operands are token-major matrices read M/N-major (64 features x 64
// tokens per box, two boxes per operand and CTA): C = U^T V reduces over tokens, and the
// epilogue adds each tile (its upper triangle, column >= row, when the problem says so) to
// an fp32 sum with atomics (Eq. 4; weight gradients).
template <bool SYRK, bool B_MN = SYRK>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(PairShape<SYRK>::THREADS, 1)
    tc_gemm_pair_kernel(const __grid_constant__ CUtensorMap map_a0, const __grid_constant__ CUtensorMap map_b0,
                        const __grid_constant__ CUtensorMap map_a1, const __grid_constant__ CUtensorMap map_b1,
                        const __grid_constant__ CUtensorMap map_c0, const __grid_constant__ CUtensorMap map_c1,
                        const PairArgs args)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* staging = smem + PAIR_STAGES * PAIR_STAGE_BYTES;   // 1024-byte aligned
    uint64_t* full = reinterpret_cast<uint64_t*>(staging + PairShape<SYRK>::STAGING);
    uint64_t* empty = full + PAIR_STAGES;
    uint64_t* tfull = empty + PAIR_STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint64_t* ring_full = drain + 1;
    uint64_t* ring_empty = ring_full + PAIR_RING;
    int* ring_item = reinterpret_cast<int*>(ring_empty + PAIR_RING);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(ring_item + PAIR_RING);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int pair = static_cast<int>(blockIdx.x >> 1);
    const int npairs = static_cast<int>(gridDim.x >> 1);

    if (threadIdx.x == 0) {
        for (int s = 0; s < PAIR_STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], 2 * 32 * PairShape<SYRK>::EPI_WARPS);   // both CTAs' epilogues
        }
        mbar_init(drain, 1);
        for (int s = 0; s < PAIR_RING; ++s) {
            mbar_init(&ring_full[s], 1);
            // the leader's MMA issuer and epilogue warps, the peer's producer and epilogue warps
            mbar_init(&ring_empty[s], 2 + 2 * PairShape<SYRK>::EPI_WARPS);
        }
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) tmem_alloc_pair(tmem_slot, PAIR_TMEM_COLS);
    if (warp == 0 && lane == 0) {
        tma_prefetch_map(&map_a0);
        tma_prefetch_map(&map_b0);
        if (args.nprob > 1) {
            tma_prefetch_map(&map_a1);
            tma_prefetch_map(&map_b1);
        }
        if (!SYRK && args.p[0].tma_store) tma_prefetch_map(&map_c0);
        if (!SYRK && args.nprob > 1 && args.p[1].tma_store) tma_prefetch_map(&map_c1);
    }
    tc_fence_before_sync();
    cluster_sync();   // barriers of both CTAs initialised before any remote arrive or copy
    tc_fence_after_sync();
    const uint32_t tmem_base = *tmem_slot;
    // The pair's MMAs write the accumulator at the leader's TMEM address in both CTAs, so
    // both allocations must have returned the same address; if not, do no work and report.
    const uint32_t peer_base = ld_shared_cluster_u32(mapa_shared(smem_u32(tmem_slot), rank ^ 1u));
    const bool tmem_agree = peer_base == tmem_base;
    if (!tmem_agree && threadIdx.x == 0) atomicExch(args.status, ESPACE_ERR_STATE);

    const int num_items =
        tmem_agree ? pair_items(args.p[0]) + (args.nprob > 1 ? pair_items(args.p[1]) : 0) : 0;
    const uint64_t limit = args.wait_limit_ns;

    // i-th work item of this pair (leader's producer only): -1 when there is none left
    auto draw = [&](int i) -> int {
        const int it = args.ticket != nullptr ? atomicAdd(args.ticket, 1) : pair + i * npairs;
        return it < num_items ? it : -1;
    };
    // the i-th item from this CTA's ring; false if the wait gave up
    auto take_item = [&](int i, int& item) -> bool {
        const int idx = i % PAIR_RING;
        if (!mbar_wait_cluster(&ring_full[idx], static_cast<uint32_t>(i / PAIR_RING) & 1u, abort_flag,
                               args.status, limit, ESPACE_ERR_TIMEOUT))
            return false;
        item = *reinterpret_cast<volatile int*>(&ring_item[idx]);
        return true;
    };
    // frees ring slot i for the leader's producer
    auto release_item = [&](int i) {
        mbar_arrive_cluster(mapa_shared(smem_u32(&ring_empty[i % PAIR_RING]), 0));
    };

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer (both CTAs)
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            int next = leader ? draw(0) : -1;
            for (int i = 0; ok; ++i) {
                int item;
                if (leader) {
                    // publish the item to both CTAs' rings once every role has taken the
                    // slot's previous one
                    const int idx = i % PAIR_RING;
                    if (!mbar_wait_cluster(&ring_empty[idx], (static_cast<uint32_t>(i / PAIR_RING) & 1u) ^ 1u,
                                           abort_flag, args.status, limit, ESPACE_ERR_TIMEOUT)) {
                        ok = false;
                        break;
                    }
                    item = next;
                    ring_item[idx] = item;
                    st_shared_cluster_u32(mapa_shared(smem_u32(&ring_item[idx]), 1), static_cast<uint32_t>(item));
                    mbar_arrive_cluster(mapa_shared(smem_u32(&ring_full[idx]), 0));
                    mbar_arrive_cluster(mapa_shared(smem_u32(&ring_full[idx]), 1));
                    if (item < 0) break;
                    next = draw(i + 1);   // its latency overlaps this item's loads
                } else {
                    if (!take_item(i, item)) {
                        ok = false;
                        break;
                    }
                    release_item(i);
                    if (item < 0) break;
                }
                int prob, tm, tn, kb0, kb1;
                pair_decode(args, item, prob, tm, tn, kb0, kb1);
                const CUtensorMap* ma = prob == 0 ? &map_a0 : &map_a1;
                const CUtensorMap* mb = prob == 0 ? &map_b0 : &map_b1;
                if (prob == 1 && args.ready != nullptr) {
                    // row block tm of A (= product 0's output) must be complete: every
                    // epilogue warp of both CTAs of every tile in it has signalled
                    const int target = 2 * (EPI_THREADS / 32) * args.p[0].tiles_n;
                    const uint64_t t0 = globaltimer_ns();
                    uint32_t spins = 0;
                    while (ld_acquire_gpu(args.ready + tm) < target) {
                        if ((++spins & 15u) == 0 && (*abort_flag || globaltimer_ns() - t0 > limit)) {
                            if (!*abort_flag) atomicExch(args.status, ESPACE_ERR_TIMEOUT);
                            *abort_flag = 1;
                            ok = false;
                            break;
                        }
                        __nanosleep(128);
                    }
                    if (!ok) break;
                    fence_proxy_async_global();   // the TMA reads below see those stores
                }
                int ak0, brow, ccol, cend;
                pair_block_of(args, prob, tn, 0, ak0, brow, ccol, cend);
                const int row_a = tm * PAIR_BM + static_cast<int>(rank) * 128;
                const int row_b = brow + static_cast<int>(rank) * 128;
                if (SYRK && args.wave_ctr != nullptr) {
                    // this pair's i-th item is in wave i (static order): wait, a bounded
                    // while, for both CTAs of every pair to have issued their wave i - 1
                    const int target = 2 * npairs * i;
                    const uint64_t g0 = globaltimer_ns();
                    while (*reinterpret_cast<volatile int*>(args.wave_ctr) < target &&
                           globaltimer_ns() - g0 < WAVE_WAIT_NS)
                        __nanosleep(256);
                }
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, args.status, limit,
                                   ESPACE_ERR_TIMEOUT)) {
                        ok = false;
                        break;
                    }
                    uint8_t* sa = smem + stage * PAIR_STAGE_BYTES;
                    uint8_t* sb = sa + PAIR_A_BYTES;
                    if (leader) mbar_arrive_expect_tx(&full[stage], 2 * PAIR_STAGE_BYTES);
                    const uint32_t bar = mapa_shared(smem_u32(&full[stage]), 0);
                    int ya = kb * BK, yb = kb * BK;
                    if (SYRK) pair_seg_rows(args, kb, ya, yb);
                    if (SYRK) {
                        // 64 features x 64 tokens per box; the second 64 features at +8 KB
                        tma_load_2d_pair(sa, ma, bar, row_a, ya);
                        tma_load_2d_pair(sa + 8192, ma, bar, row_a + 64, ya);
                    } else {
                        tma_load_2d_pair(sa, ma, bar, ak0 + kb * BK, row_a);
                    }
                    if (B_MN) {
                        tma_load_2d_pair(sb, mb, bar, row_b, yb);
                        tma_load_2d_pair(sb + 8192, mb, bar, row_b + 64, yb);
                    } else {
                        tma_load_2d_pair(sb, mb, bar, kb * BK, row_b);
                    }
                    if (++stage == PAIR_STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (SYRK && args.wave_ctr != nullptr) atomicAdd(args.wave_ctr, 1);
            }
            if (!ok) settle_copies();
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (leader)
        if (lane == 0 && leader) {
            static_assert(!SYRK || B_MN, "token-reduction programs read both operands M/N-major");
            constexpr uint32_t idesc = idesc_bf16_f32(PAIR_BM, PAIR_BN, SYRK, B_MN);
            // K-major: the next 16-element K slice starts 32 bytes along the swizzled row;
            // M/N-major: 16 tokens further = 16 rows of 128 bytes, 64-feature atoms 8 KB apart
            constexpr uint32_t a_step = SYRK ? 2048u : 32u, a_lbo = SYRK ? 8192u : 16u;
            constexpr uint32_t b_step = B_MN ? 2048u : 32u, b_lbo = B_MN ? 8192u : 16u;
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int i = 0; ok; ++i) {
                int item;
                if (!take_item(i, item)) break;
                release_item(i);
                if (item < 0) break;
                int prob, tm, tn, kb0, kb1;
                pair_decode(args, item, prob, tm, tn, kb0, kb1);
                // one accumulation per item, or per 16-block chunk of it for SYRK
                const int chunk = SYRK ? SYRK_CHUNK : (kb1 - kb0);
                for (int c0 = kb0; ok && c0 < kb1; c0 += chunk) {
                    const int c1 = min(c0 + chunk, kb1);
                    if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, args.status, limit,
                                   ESPACE_ERR_TIMEOUT)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after_sync();
                    const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * PAIR_BN);
                    for (int kb = c0; kb < c1; ++kb) {
                        if (!mbar_wait(&full[stage], phase, abort_flag, args.status, limit,
                                       ESPACE_ERR_TIMEOUT)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after_sync();
                        const uint32_t a_addr = smem_u32(smem + stage * PAIR_STAGE_BYTES);
                        const uint32_t b_addr = a_addr + PAIR_A_BYTES;
#pragma unroll
                        for (int j = 0; j < BK / UMMA_K; ++j) {
                            const uint64_t ad = smem_desc_sw128(a_addr + j * a_step, a_lbo, 1024);
                            const uint64_t bd = smem_desc_sw128(b_addr + j * b_step, b_lbo, 1024);
                            umma_bf16_pair(d_tmem, ad, bd, idesc, (kb > c0 || j > 0) ? 1u : 0u);
                        }
                        umma_commit_pair(&empty[stage], 0x3);   // frees the stage in both CTAs
                        if (++stage == PAIR_STAGES) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                    if (!ok) break;
                    umma_commit_pair(&tfull[acc], 0x3);          // both halves ready to drain
                    if (++acc == PAIR_ACCS) {
                        acc = 0;
                        acc_phase ^= 1u;
                    }
                }
            }
            umma_commit_pair(drain, 0x1);
            volatile int never = 0;
            mbar_wait(drain, 0, &never, args.status, cleanup_limit(limit), ESPACE_ERR_TIMEOUT);
        }
    } else if (SYRK) {
        // ------------------------------------------------------------ SYRK epilogue (8 warps)
        // warp pair (w, w + 4) shares a TMEM lane quarter and splits its 256 columns
        const int ew = warp - 2;
        const int quarter = warp & 3;
        const int half = ew >> 2;
        const int row_in_tile = static_cast<int>(rank) * 128 + quarter * 32 + lane;
        int acc = 0;
        uint32_t acc_phase = 0;
        bool ok = true;
        for (int i = 0; ok; ++i) {
            int item;
            if (!take_item(i, item)) break;
            __syncwarp();
            if (lane == 0) release_item(i);
            if (item < 0) break;
            int prob, tm, tn, kb0, kb1;
            pair_decode(args, item, prob, tm, tn, kb0, kb1);
            const PairProblem pb = pair_problem_of(args, prob);
            float run[128];
#pragma unroll
            for (int i = 0; i < 128; ++i) run[i] = 0.f;
            for (int c0 = kb0; c0 < kb1; c0 += SYRK_CHUNK) {
                if (!mbar_wait(&tfull[acc], acc_phase, abort_flag, args.status, limit,
                               ESPACE_ERR_TIMEOUT)) {
                    ok = false;
                    break;
                }
                tc_fence_after_sync();
                const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                                       static_cast<uint32_t>(acc * PAIR_BN + half * 128);
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    uint32_t v[16];
                    tmem_ld_16cols(t_row + static_cast<uint32_t>(c * 16), v);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 16; ++i) run[c * 16 + i] += __uint_as_float(v[i]);
                }
                tc_fence_before_sync();
                mbar_arrive_cluster(mapa_shared(smem_u32(&tempty[acc]), 0));
                if (++acc == PAIR_ACCS) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
            }
            if (!ok) break;
            // S[row][col] += run, or = run for a program that assigns (for col >= row only
            // when the problem is a triangle), 16 bytes at a time
            const int row = tm * PAIR_BM + row_in_tile;
            if (row < pb.rows) {
                float* s_row = reinterpret_cast<float*>(pb.out) + static_cast<int64_t>(row) * pb.ldo;
                const int colb = tn * PAIR_BN + half * 128;
                const int cmin = (pb.upper & 1) ? row : 0;
                if (pb.upper & 2) {
#pragma unroll
                    for (int i = 0; i < 128; i += 4) {
                        const int col = colb + i;
                        if (col >= cmin && col + 3 < pb.cols) {
                            *reinterpret_cast<float4*>(s_row + col) =
                                make_float4(run[i], run[i + 1], run[i + 2], run[i + 3]);
                        } else {
#pragma unroll
                            for (int j = 0; j < 4; ++j)
                                if (col + j >= cmin && col + j < pb.cols) s_row[col + j] = run[i + j];
                        }
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < 128; i += 4) {
                        const int col = colb + i;
                        if (col >= cmin && col + 3 < pb.cols) {
                            atomicAdd(reinterpret_cast<float4*>(s_row + col),
                                      make_float4(run[i], run[i + 1], run[i + 2], run[i + 3]));
                        } else {
#pragma unroll
                            for (int j = 0; j < 4; ++j)
                                if (col + j >= cmin && col + j < pb.cols) atomicAdd(s_row + col + j, run[i + j]);
                        }
                    }
                }
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue (both CTAs)
        const int quarter = warp & 3;
        const int row_in_tile = static_cast<int>(rank) * 128 + quarter * 32 + lane;
        // this warp's two staging buffers (32 rows x 128 bytes each, swizzled as the map's box)
        uint8_t* stage_buf = staging + quarter * 2 * PAIR_EPI_BUF;
        uint32_t chunks = 0;   // slices this warp has handed to TMA (buffer = chunks & 1)
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int i = 0;; ++i) {
            int item;
            if (!take_item(i, item)) break;
            __syncwarp();
            if (lane == 0) release_item(i);
            if (item < 0) break;
            int prob, tm, tn, kb0, kb1;
            pair_decode(args, item, prob, tm, tn, kb0, kb1);
            const PairProblem pb = pair_problem_of(args, prob);
            if (!mbar_wait(&tfull[acc], acc_phase, abort_flag, args.status, limit,
                           ESPACE_ERR_TIMEOUT))
                break;
            tc_fence_after_sync();
            const int row = tm * PAIR_BM + row_in_tile;
            const uint32_t t_row = tmem_base + (static_cast<uint32_t>(quarter * 32) << 16) +
                                   static_cast<uint32_t>(acc * PAIR_BN);
            int ak0, brow, ccol, cend;
            pair_block_of(args, prob, tn, pb.cols, ak0, brow, ccol, cend);
            if (pb.tma_store) {
                // 64-column slices: TMEM -> registers -> bf16 in the staging buffer (16-byte
                // chunk c of row r at chunk c ^ (r % 8)) -> one TMA store per slice, clipped
                // at the tensor's last row and column
                const CUtensorMap* mc = prob == 0 ? &map_c0 : &map_c1;
                const int y0 = tm * PAIR_BM + static_cast<int>(rank) * 128 + quarter * 32;
#pragma unroll 1
                for (int c = 0; c < PAIR_BN; c += 64) {
                    const int col0 = ccol + c;
                    if (col0 >= cend) break;             // uniform across the warp
                    uint8_t* buf = stage_buf + (chunks & 1u) * PAIR_EPI_BUF;
                    if (chunks >= 2) {
                        // the store that used this buffer two slices ago has read it
                        if (lane == 0) bulk_wait_group_read<1>();
                        __syncwarp();
                    }
                    uint32_t v[32];
                    const uint32_t row_addr = smem_u32(buf) + static_cast<uint32_t>(lane) * 128u;
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        tmem_ld_32cols(t_row + static_cast<uint32_t>(c + 32 * h), v);
                        tmem_ld_wait();
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            uint4 w;
                            w.x = pack_bf16x2(__uint_as_float(v[8 * q + 0]), __uint_as_float(v[8 * q + 1]));
                            w.y = pack_bf16x2(__uint_as_float(v[8 * q + 2]), __uint_as_float(v[8 * q + 3]));
                            w.z = pack_bf16x2(__uint_as_float(v[8 * q + 4]), __uint_as_float(v[8 * q + 5]));
                            w.w = pack_bf16x2(__uint_as_float(v[8 * q + 6]), __uint_as_float(v[8 * q + 7]));
                            const uint32_t chunk = static_cast<uint32_t>((4 * h + q) ^ (lane & 7));
                            st_shared_v4(row_addr + chunk * 16u, w);
                        }
                    }
                    fence_proxy_async_shared();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_2d(mc, buf, col0, y0);
                        bulk_commit_group();
                    }
                    ++chunks;
                }
            } else {
#pragma unroll 1
                for (int c = 0; c < PAIR_BN; c += 32) {
                    const int col0 = ccol + c;
                    if (col0 >= cend) break;             // uniform across the warp
                    uint32_t v[32];
                    tmem_ld_32cols(t_row + static_cast<uint32_t>(c), v);
                    tmem_ld_wait();
                    if (row >= pb.rows) continue;
                    __nv_bfloat16* out_row =
                        reinterpret_cast<__nv_bfloat16*>(pb.out) + static_cast<int64_t>(row) * pb.ldo;
                    if (col0 + 32 <= cend) {
                        uint4* dst = reinterpret_cast<uint4*>(out_row + col0);
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            uint4 q;
                            q.x = pack_bf16x2(__uint_as_float(v[8 * i + 0]), __uint_as_float(v[8 * i + 1]));
                            q.y = pack_bf16x2(__uint_as_float(v[8 * i + 2]), __uint_as_float(v[8 * i + 3]));
                            q.z = pack_bf16x2(__uint_as_float(v[8 * i + 4]), __uint_as_float(v[8 * i + 5]));
                            q.w = pack_bf16x2(__uint_as_float(v[8 * i + 6]), __uint_as_float(v[8 * i + 7]));
                            dst[i] = q;
                        }
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (col0 + i < cend)
                                out_row[col0 + i] = __float2bfloat16_rn(__uint_as_float(v[i]));
                    }
                }
            }
            tc_fence_before_sync();
            mbar_arrive_cluster(mapa_shared(smem_u32(&tempty[acc]), 0));
            if (++acc == PAIR_ACCS) {
                acc = 0;
                acc_phase ^= 1u;
            }
            if (prob == 0 && args.nprob > 1 && args.ready != nullptr) {
                // publish this warp's 32 rows of the tile to the second product's producers
                // (per warp, so that no block-wide barrier can wait on a warp that gave up);
                // TMA stores must have completed, not only read their source
                if (pb.tma_store && lane == 0) bulk_wait_group<0>();
                fence_proxy_async_global();
                __threadfence();
                __syncwarp();
                if (lane == 0) red_release_gpu_add(args.ready + tm, 1);
            }
        }
        // every TMA store of this warp has completed before its staging can go away
        if (lane == 0) bulk_wait_group<0>();
    }

    __syncwarp();
    // a CTA whose roles gave up may still have copies in flight, into its own shared memory
    // or signalling its peer's barriers: both CTAs stay until they have landed
    if (threadIdx.x == 0 && *abort_flag) settle_copies();
    tc_fence_before_sync();
    cluster_sync();   // no CTA leaves while its peer may still touch its barriers or TMEM
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc_pair(tmem_base, PAIR_TMEM_COLS);
    }
    if (args.exit_ctr != nullptr && threadIdx.x == 0) {
        // every thread of this CTA is past its last use of the counters (cluster barrier);
        // the last CTA of the grid zeroes them for the next launch
        __threadfence();
        if (atomicAdd(args.exit_ctr, 1) == static_cast<int>(gridDim.x) - 1) {
            __threadfence();
            volatile int* r = args.ready;
            for (int b = 0; b < args.nready; ++b) r[b] = 0;
            if (args.ticket != nullptr) *reinterpret_cast<volatile int*>(args.ticket) = 0;
            if (args.wave_ctr != nullptr) *reinterpret_cast<volatile int*>(args.wave_ctr) = 0;
            __threadfence();
            *reinterpret_cast<volatile int*>(args.exit_ctr) = 0;
        }
    }
}

// =========================================================================== host side

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// 2-D bf16 tensor [outer][inner] with a row pitch of `pitch_elems`, 128-byte swizzled boxes
// of box_inner x box_outer elements, zero fill outside the tensor.
bool encode_map(CUtensorMap* map, const void* base, uint64_t inner, uint64_t outer,
                uint64_t pitch_elems, uint32_t box_inner, uint32_t box_outer)
{
    EncodeTiledFn fn = encode_fn();
    if (fn == nullptr) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {pitch_elems * 2};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, int STAGES, bool MN_MAJOR, int EPI>
cudaError_t launch_kernel(const CUtensorMap& ma, const CUtensorMap& mb, const TcGemmArgs& args,
                          int grid, cudaStream_t stream)
{
    using Cfg = TcCfg<BN, STAGES>;
    auto kern = tc_gemm_kernel<BN, STAGES, MN_MAJOR, EPI>;
    // per instantiation and device; a race only repeats the idempotent call
    static std::atomic<bool> attr_set[64];   // per device; a repeated set is harmless
    int device = 0;
    cudaGetDevice(&device);
    if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
    if (!attr_set[device].load(std::memory_order_acquire)) {
        cudaError_t e =
            cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set[device].store(true, std::memory_order_release);
    }
    if (args.pdl) {
        // may start while the preceding grid on the stream finishes (see TcGemmArgs::pdl)
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(grid);
        cfg.blockDim = dim3(GEMM_THREADS);
        cfg.dynamicSmemBytes = Cfg::SMEM_BYTES;
        cfg.stream = stream;
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        return cudaLaunchKernelEx(&cfg, kern, ma, mb, args);
    }
    kern<<<grid, GEMM_THREADS, Cfg::SMEM_BYTES, stream>>>(ma, mb, args);
    return cudaGetLastError();
}

PairProblem pair_problem(int rows, int cols, int kdim, void* out, int64_t ldo)
{
    PairProblem p{};
    p.rows = rows;
    p.cols = cols;
    p.kblocks = (kdim + BK - 1) / BK;
    p.tiles_n = (cols + PAIR_BN - 1) / PAIR_BN;
    p.num_tiles = ((rows + PAIR_BM - 1) / PAIR_BM) * p.tiles_n;
    p.ksplit = 1;
    p.kb_per_split = p.kblocks;
    p.tile_list = nullptr;
    p.out = out;
    p.ldo = ldo;
    return p;
}

template <bool SYRK, bool B_MN = SYRK>
cudaError_t launch_pair(const CUtensorMap* maps, PairArgs& a, const DeviceInfo* dev, cudaStream_t stream)
{
    const int items = a.p[0].num_tiles * a.p[0].ksplit + (a.nprob > 1 ? a.p[1].num_tiles * a.p[1].ksplit : 0);
    const int pairs = std::min(items, dev->num_sms / 2);
    auto kern = tc_gemm_pair_kernel<SYRK, B_MN>;
    constexpr int smem = PairShape<SYRK>::SMEM_BYTES;
    static std::atomic<bool> attr_set[64];   // per device; a repeated set is harmless
    if (dev->device < 0 || dev->device >= 64) return cudaErrorInvalidDevice;
    if (!attr_set[dev->device].load(std::memory_order_acquire)) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        attr_set[dev->device].store(true, std::memory_order_release);
    }
    // output tensor maps of the bf16 programs (TMA stores); a problem whose output cannot
    // be described to TMA (pitch not a multiple of 16 bytes, base not 16-byte aligned) or
    // that stores only part of its columns (block-diagonal) keeps the direct stores
    CUtensorMap cmaps[2];
    memset(cmaps, 0, sizeof(cmaps));
    for (int q = 0; q < a.nprob && !SYRK; ++q) {
        PairProblem& pq = a.p[q];
        pq.tma_store = 0;
        if (a.nblocks == 0 && pq.cols >= 64 && pq.rows >= 32 && pq.ldo % 8 == 0 &&
            (reinterpret_cast<uintptr_t>(pq.out) & 15u) == 0 &&
            encode_map(&cmaps[q], pq.out, pq.cols, pq.rows, pq.ldo, 64, 32))
            pq.tma_store = 1;
    }
    if (a.nprob < 2) cmaps[1] = cmaps[0];
    kern<<<2 * pairs, PairShape<SYRK>::THREADS, smem, stream>>>(maps[0], maps[1], maps[2], maps[3], cmaps[0],
                                                                  cmaps[1], a);
    return cudaGetLastError();
}

// 256 x 256 tiles on CTA pairs; grid = 2 x min(tiles, SMs / 2).
cudaError_t launch_gemm_tn_pair(const void* A, int64_t lda, const void* B, int64_t ldb, int rows,
                                int cols, int kdim, void* C, int64_t ldc, cudaStream_t stream,
                                const DeviceInfo* dev)
{
    CUtensorMap maps[4];
    if (!encode_map(&maps[0], A, kdim, rows, lda, BK, 128)) return cudaErrorInvalidValue;
    if (!encode_map(&maps[1], B, kdim, cols, ldb, BK, 128)) return cudaErrorInvalidValue;
    maps[2] = maps[0];
    maps[3] = maps[1];
    PairArgs a{};
    a.p[0] = pair_problem(rows, cols, kdim, C, ldc);
    a.nprob = 1;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_pair<false>(maps, a, dev, stream);
}

}  // namespace

cudaError_t launch_gemm_tn_blocks(const void* A, int64_t lda, int a_cols, const void* B, int rows, int nblocks,
                                  const int* ak0, const int* c0, const int* cw, int kdim, void* C, int64_t ldc,
                                  cudaStream_t stream)
{
    if (rows <= 0) return cudaSuccess;
    if (nblocks < 1 || nblocks > PAIR_MAX_BLOCKS || kdim <= 0 || kdim % BK != 0) return cudaErrorInvalidValue;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    if (dev->num_sms < 2) return cudaErrorInvalidConfiguration;
    PairArgs a{};
    int cols = 0, tiles = 0;
    for (int g = 0; g < nblocks; ++g) {
        if (cw[g] <= 0 || c0[g] != cols || ak0[g] < 0 || ak0[g] % BK != 0 || ak0[g] + kdim > a_cols)
            return cudaErrorInvalidValue;
        a.tile0[g] = tiles;
        a.ak0[g] = ak0[g];
        a.c0[g] = c0[g];
        a.cw[g] = cw[g];
        tiles += (cw[g] + PAIR_BN - 1) / PAIR_BN;
        cols += cw[g];
    }
    a.tile0[nblocks] = tiles;
    a.nblocks = nblocks;
    CUtensorMap maps[4];
    if (!encode_map(&maps[0], A, a_cols, rows, lda, BK, 128)) return cudaErrorInvalidValue;
    if (!encode_map(&maps[1], B, kdim, cols, kdim, BK, 128)) return cudaErrorInvalidValue;
    maps[2] = maps[0];
    maps[3] = maps[1];
    a.p[0] = pair_problem(rows, cols, kdim, C, ldc);
    a.p[0].tiles_n = tiles;
    a.p[0].num_tiles = ((rows + PAIR_BM - 1) / PAIR_BM) * tiles;
    a.nprob = 1;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_pair<false>(maps, a, dev, stream);
}

// The CTA-pair kernel is used unless ESPACE_DISABLE_PAIR_GEMM=1 is set in the environment.
bool pair_kernel_enabled()
{
    static const bool enabled = [] {
        const char* v = getenv("ESPACE_DISABLE_PAIR_GEMM");
        return !(v != nullptr && v[0] == '1');
    }();
    return enabled;
}

cudaError_t launch_gemm_tn(const void* A, int64_t lda, const void* B, int64_t ldb, int rows,
                           int cols, int kdim, void* C, int64_t ldc, cudaStream_t stream)
{
    if (rows <= 0 || cols <= 0) return cudaSuccess;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    if (rows > 128 && cols > 128 && dev->num_sms >= 2 && pair_kernel_enabled())
        return launch_gemm_tn_pair(A, lda, B, ldb, rows, cols, kdim, C, ldc, stream, dev);
    const bool wide = cols > 128;
    const int bn = wide ? 256 : 128;
    CUtensorMap ma, mb;
    if (!encode_map(&ma, A, kdim, rows, lda, BK, BM)) return cudaErrorInvalidValue;
    if (!encode_map(&mb, B, kdim, cols, ldb, BK, bn)) return cudaErrorInvalidValue;
    TcGemmArgs a{};
    a.rows = rows;
    a.cols = cols;
    a.kblocks = (kdim + BK - 1) / BK;
    a.tiles_n = (cols + bn - 1) / bn;
    a.num_tiles = ((rows + BM - 1) / BM) * a.tiles_n;
    a.ksplit = 1;
    a.kb_per_split = a.kblocks;
    a.tile_list = nullptr;
    a.out = C;
    a.ldo = ldc;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    const int grid = std::min(a.num_tiles, dev->num_sms);
    if (wide) return launch_kernel<256, 4, false, EPI_STORE_BF16>(ma, mb, a, grid, stream);
    return launch_kernel<128, 6, false, EPI_STORE_BF16>(ma, mb, a, grid, stream);
}

// Swapped product for few tokens: tiles of 128 weight rows x 128 (ntok <= 128) or 256
// tokens. When the tiles would leave more than half of the SMs idle, the reduction splits
// over CTAs: about one work item per SM, at least 4 k-blocks per split.
SwapPlan gemm_swap_plan(int rows, int ntok, int kdim, int num_sms, bool allow_split)
{
    SwapPlan pl;
    pl.bn = ntok <= 128 ? 128 : 256;
    pl.tiles = ((rows + BM - 1) / BM) * ((ntok + pl.bn - 1) / pl.bn);
    pl.kblocks = (kdim + BK - 1) / BK;
    pl.ksplit = 1;
    pl.kb_per_split = pl.kblocks;
    if (allow_split && pl.tiles < num_sms / 2) {
        const int want = std::max(1, num_sms / pl.tiles);
        pl.kb_per_split = std::min(pl.kblocks, std::max(4, (pl.kblocks + want - 1) / want));
        pl.ksplit = (pl.kblocks + pl.kb_per_split - 1) / pl.kb_per_split;
    }
    pl.ld_part = (ntok + 31) / 32 * 32;
    pl.part_elems = pl.ksplit > 1 ? static_cast<int64_t>(pl.ksplit) * rows * pl.ld_part : 0;
    return pl;
}

// out[n][r] = bf16(sum over s, in order, of part[(s * rows + r) * ld_part + n]). A block of
// 32 x 32 threads takes 32 rows x 32 tokens, one output each: the partials are read along
// tokens and the bf16 results written along rows, both coalesced, through shared memory.
__global__ void __launch_bounds__(1024) reduce_splits_kernel(const float* __restrict__ part, int ksplit, int rows,
                                                             int64_t ld_part, int ntok, __nv_bfloat16* __restrict__ out,
                                                             int64_t ldo, int pdl)
{
    __shared__ float tile[32][33];
    if (pdl) {
        // launched early: let the next grid start its own weight loads, then wait for the
        // partials of the preceding one
        if (threadIdx.x == 0) grid_dep_launch_dependents();
        grid_dep_wait();
    }
    const int r0 = blockIdx.x * 32, n0 = blockIdx.y * 32;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    float acc = 0.f;
    if (r0 + ty < rows) {
        const float* src = part + static_cast<int64_t>(r0 + ty) * ld_part + n0 + tx;
        const int64_t step = static_cast<int64_t>(rows) * ld_part;
        // four partials in flight at a time, added in split order
        int sp = 0;
        for (; sp + 4 <= ksplit; sp += 4) {
            const float a0 = __ldcg(src + sp * step), a1 = __ldcg(src + (sp + 1) * step);
            const float a2 = __ldcg(src + (sp + 2) * step), a3 = __ldcg(src + (sp + 3) * step);
            acc += a0;
            acc += a1;
            acc += a2;
            acc += a3;
        }
        for (; sp < ksplit; ++sp) acc += __ldcg(src + sp * step);
    }
    tile[ty][tx] = acc;
    __syncthreads();
    const int n = n0 + ty, r = r0 + tx;
    if (n < ntok && r < rows) out[static_cast<int64_t>(n) * ldo + r] = __float2bfloat16_rn(tile[tx][ty]);
}

cudaError_t launch_gemm_swap(const void* W, int64_t ldw, const void* X, int64_t ldx, int rows, int ntok, int kdim,
                             void* out, int64_t ldo, float* part, cudaStream_t stream, bool pdl)
{
    if (rows <= 0 || ntok <= 0) return cudaSuccess;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    // without a workspace the reduction is not split
    const SwapPlan pl = gemm_swap_plan(rows, ntok, kdim, dev->num_sms, part != nullptr);
    // token tiles load only the rows that exist (rounded up to 8)
    const int b_rows = std::min(pl.bn, (ntok + 7) / 8 * 8);
    CUtensorMap ma, mb;
    if (!encode_map(&ma, W, kdim, rows, ldw, BK, BM)) return cudaErrorInvalidValue;
    if (!encode_map(&mb, X, kdim, ntok, ldx, BK, b_rows)) return cudaErrorInvalidValue;
    TcGemmArgs a{};
    a.rows = rows;
    a.cols = ntok;
    a.kblocks = pl.kblocks;
    a.tiles_n = (ntok + pl.bn - 1) / pl.bn;
    a.num_tiles = pl.tiles;
    a.ksplit = pl.ksplit;
    a.kb_per_split = pl.kb_per_split;
    a.tile_list = nullptr;
    a.out = out;
    a.ldo = ldo;
    a.part = part;
    a.ld_part = pl.ld_part;
    a.b_rows = b_rows;
    a.pdl = pdl ? 1 : 0;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    const int grid = std::min(pl.tiles * pl.ksplit, dev->num_sms);
    if (pl.ksplit > 1) {
        cudaError_t e = pl.bn == 128 ? launch_kernel<128, 6, false, EPI_SPLIT_BF16_T>(ma, mb, a, grid, stream)
                                     : launch_kernel<256, 4, false, EPI_SPLIT_BF16_T>(ma, mb, a, grid, stream);
        if (e != cudaSuccess) return e;
        const dim3 grid_r((rows + 31) / 32, (ntok + 31) / 32);
        if (pdl) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = grid_r;
            cfg.blockDim = dim3(1024);
            cfg.dynamicSmemBytes = 0;
            cfg.stream = stream;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
            attr[0].val.programmaticStreamSerializationAllowed = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            return cudaLaunchKernelEx(&cfg, reduce_splits_kernel, static_cast<const float*>(part), pl.ksplit, rows,
                                      pl.ld_part, ntok, static_cast<__nv_bfloat16*>(out), ldo, 1);
        }
        reduce_splits_kernel<<<grid_r, 1024, 0, stream>>>(part, pl.ksplit, rows, pl.ld_part, ntok,
                                                         static_cast<__nv_bfloat16*>(out), ldo, 0);
        return cudaGetLastError();
    }
    if (pl.bn == 128) return launch_kernel<128, 6, false, EPI_STORE_BF16_T>(ma, mb, a, grid, stream);
    return launch_kernel<256, 4, false, EPI_STORE_BF16_T>(ma, mb, a, grid, stream);
}

namespace {

struct TileList {
    int K = -1;
    int2* dev = nullptr;
    int count = 0;
};

// Upper-triangle tile pairs for one K and tile shape (rows x cols), kept per device.
int2* syrk_tiles(int K, int tile_rows, int tile_cols, int* count)
{
    static std::mutex mu;
    struct Entry {
        int device, K, tr, tc;
        TileList list;
    };
    static std::vector<Entry> cache;
    int device = 0;
    cudaGetDevice(&device);
    std::lock_guard<std::mutex> lock(mu);
    for (auto& e : cache)
        if (e.device == device && e.K == K && e.tr == tile_rows && e.tc == tile_cols) {
            *count = e.list.count;
            return e.list.dev;
        }
    // Z order (bit-interleaved tile row and column): the workers take consecutive items
    // together and stream the tokens at about the same pace, so items that run at the same
    // time should share feature slices. Any run of consecutive tiles in Z order is compact:
    // a wave of 76 CTA pairs reads ~23 distinct 256-feature slices of the token window at
    // K = 24576 instead of ~60 in row-major order, which keeps them in L2.
    std::vector<int2> host;
    const int tm_n = (K + tile_rows - 1) / tile_rows, tn_n = (K + tile_cols - 1) / tile_cols;
    for (int tm = 0; tm < tm_n; ++tm)
        for (int tn = 0; tn < tn_n; ++tn)
            if (tn * tile_cols + tile_cols - 1 >= tm * tile_rows) host.push_back(make_int2(tm, tn));
    auto morton = [](int2 t) {
        uint64_t r = 0;
        for (int b = 0; b < 16; ++b)
            r |= ((static_cast<uint64_t>(t.x) >> b) & 1u) << (2 * b + 1) |
                 ((static_cast<uint64_t>(t.y) >> b) & 1u) << (2 * b);
        return r;
    };
    std::stable_sort(host.begin(), host.end(), [&](int2 a, int2 b) { return morton(a) < morton(b); });
    int2* dev = nullptr;
    if (cudaMalloc(&dev, host.size() * sizeof(int2)) != cudaSuccess) return nullptr;
    if (cudaMemcpy(dev, host.data(), host.size() * sizeof(int2), cudaMemcpyHostToDevice) != cudaSuccess) {
        cudaFree(dev);
        return nullptr;
    }
    Entry e;
    e.device = device;
    e.K = K;
    e.tr = tile_rows;
    e.tc = tile_cols;
    e.list.K = K;
    e.list.dev = dev;
    e.list.count = static_cast<int>(host.size());
    cache.push_back(e);
    *count = e.list.count;
    return dev;
}

// Token splits per tile: the count s that minimises the last worker's time, ceil(tiles s /
// workers) waves of ceil(kblocks / s) k-blocks plus a per-item cost of item_kb k-blocks of
// MMA (the atomic adds of a 256 x 256 fp32 tile and the item's pipeline fill), with at least
// 16 k-blocks (1024 tokens) per split; more splits are taken only for a modelled gain of 2%
// or more. The per-item cost is the caller's, measured for its kind of launch.
void choose_splits(int kblocks, int tiles, int workers, int64_t item_kb, int* ksplit, int* kb_per_split)
{
    int best_s = 1;
    int64_t best = INT64_MAX;
    for (int s = 1; s <= 64; ++s) {
        const int kbps = (kblocks + s - 1) / s;
        if (s > 1 && kbps < 16) break;
        if ((kblocks + kbps - 1) / kbps != s) continue;   // the same split as a smaller s
        const int64_t waves = (static_cast<int64_t>(tiles) * s + workers - 1) / workers;
        const int64_t cost = waves * (kbps + item_kb);
        if (cost * 50 < best * 49) {
            best = cost;
            best_s = s;
        }
    }
    *ksplit = best_s;
    *kb_per_split = (kblocks + best_s - 1) / best_s;
}

}  // namespace

cudaError_t launch_syrk_upper(const void* X, int64_t N, int K, float* S, cudaStream_t stream, int* sched)
{
    return launch_syrk_cross_upper(X, X, N, K, S, stream, sched);
}

cudaError_t launch_syrk_upper_two(const void* X, const void* Y, int64_t N, int K, float* Sx, float* Sy,
                                  bool assign, cudaStream_t stream)
{
    if (N <= 0) return cudaSuccess;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    const int kblocks = static_cast<int>((N + BK - 1) / BK);
    int ksplit = 1, kbps = kblocks;
    const bool pair = K > 128 && dev->num_sms >= 2 && pair_kernel_enabled();
    if (pair) {
        int count = 0;
        if (syrk_tiles(K, PAIR_BM, PAIR_BN, &count) == nullptr) return cudaErrorMemoryAllocation;
        choose_splits(kblocks, 2 * count, dev->num_sms / 2, 8, &ksplit, &kbps);
    }
    if (assign && (!pair || ksplit > 1)) {
        // split reductions add: start from zero
        const int64_t kk = static_cast<int64_t>(K) * K;
        cudaError_t e = launch_zero_f32(Sx, kk, stream);
        if (e == cudaSuccess) e = launch_zero_f32(Sy, kk, stream);
        if (e != cudaSuccess) return e;
    }
    if (!pair) {
        cudaError_t e = launch_syrk_upper(X, N, K, Sx, stream);
        return e != cudaSuccess ? e : launch_syrk_upper(Y, N, K, Sy, stream);
    }
    int count = 0;
    const int2* tiles = syrk_tiles(K, PAIR_BM, PAIR_BN, &count);
    if (tiles == nullptr) return cudaErrorMemoryAllocation;
    CUtensorMap maps[4];
    if (!encode_map(&maps[0], X, K, static_cast<uint64_t>(N), K, 64, BK)) return cudaErrorInvalidValue;
    if (!encode_map(&maps[2], Y, K, static_cast<uint64_t>(N), K, 64, BK)) return cudaErrorInvalidValue;
    maps[1] = maps[0];
    maps[3] = maps[2];
    PairArgs a{};
    float* outs[2] = {Sx, Sy};
    for (int q = 0; q < 2; ++q) {
        PairProblem& p = a.p[q];
        p.rows = K;
        p.cols = K;
        p.kblocks = kblocks;
        p.tiles_n = 0;
        p.num_tiles = count;
        p.ksplit = ksplit;
        p.kb_per_split = kbps;
        p.tile_list = tiles;
        p.out = outs[q];
        p.ldo = K;
        p.upper = assign && ksplit == 1 ? 3 : 1;
    }
    a.nprob = 2;       // independent problems: no ready counters
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_pair<true>(maps, a, dev, stream);
}

cudaError_t launch_syrk_segments_upper(const void* Q, int64_t q_rows, int K, int seg_rows, int nseg,
                                       const int* seg_u, const int* seg_v, float* S, cudaStream_t stream)
{
    if (nseg <= 0) return cudaSuccess;
    if (nseg > PAIR_MAX_SEGS || seg_rows <= 0 || seg_rows % BK != 0 || K <= 0) return cudaErrorInvalidValue;
    for (int q = 0; q < nseg; ++q)
        if (seg_u[q] < 0 || seg_v[q] < 0 || seg_u[q] % BK != 0 || seg_v[q] % BK != 0 ||
            seg_u[q] + seg_rows > q_rows || seg_v[q] + seg_rows > q_rows)
            return cudaErrorInvalidValue;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    if (K <= 128 || dev->num_sms < 2 || !pair_kernel_enabled()) {
        // one two-operand SYRK per segment
        const size_t ld = static_cast<size_t>(K);
        for (int q = 0; q < nseg; ++q) {
            const auto* base = static_cast<const uint16_t*>(Q);
            cudaError_t e = launch_syrk_cross_upper(base + seg_u[q] * ld, base + seg_v[q] * ld, seg_rows, K, S, stream);
            if (e != cudaSuccess) return e;
        }
        return cudaSuccess;
    }
    int count = 0;
    const int2* tiles = syrk_tiles(K, PAIR_BM, PAIR_BN, &count);
    if (tiles == nullptr) return cudaErrorMemoryAllocation;
    CUtensorMap maps[4];
    if (!encode_map(&maps[0], Q, K, static_cast<uint64_t>(q_rows), K, 64, BK)) return cudaErrorInvalidValue;
    maps[1] = maps[2] = maps[3] = maps[0];
    PairArgs a{};
    PairProblem& p = a.p[0];
    p.rows = K;
    p.cols = K;
    p.kblocks = nseg * (seg_rows / BK);
    p.tiles_n = 0;
    p.num_tiles = count;
    // (8 k-blocks per item: five splits of the NL-MSE products at K = 4096 measured 498 us a
    // call, one split 512 us)
    choose_splits(p.kblocks, count, dev->num_sms / 2, 8, &p.ksplit, &p.kb_per_split);
    p.tile_list = tiles;
    p.out = S;
    p.ldo = K;
    p.upper = 1;
    a.nprob = 1;
    a.seg_n = nseg;
    for (int q = 0; q < nseg; ++q) {
        a.seg_a[q] = seg_u[q];
        a.seg_b[q] = seg_v[q];
    }
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_pair<true>(maps, a, dev, stream);
}

cudaError_t launch_syrk_cross_upper(const void* X, const void* Y, int64_t N, int K, float* S, cudaStream_t stream,
                                    int* sched)
{
    if (N <= 0) return cudaSuccess;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    const int kblocks = static_cast<int>((N + BK - 1) / BK);
    if (K > 128 && dev->num_sms >= 2 && pair_kernel_enabled()) {
        // 256 x 256 upper-triangle tiles on CTA pairs
        int count = 0;
        const int2* tiles = syrk_tiles(K, PAIR_BM, PAIR_BN, &count);
        if (tiles == nullptr) return cudaErrorMemoryAllocation;
        CUtensorMap maps[4];
        if (!encode_map(&maps[0], X, K, static_cast<uint64_t>(N), K, 64, BK)) return cudaErrorInvalidValue;
        if (!encode_map(&maps[1], Y, K, static_cast<uint64_t>(N), K, 64, BK)) return cudaErrorInvalidValue;
        maps[2] = maps[0];
        maps[3] = maps[1];
        PairArgs a{};
        PairProblem& p = a.p[0];
        p.rows = K;
        p.cols = K;
        p.kblocks = kblocks;
        p.tiles_n = 0;
        p.num_tiles = count;
        // (24 k-blocks per item: at K = 4096 over 65,536 tokens one split measured 0.670 ms,
        // the five that 8 k-blocks per item pick 0.685 ms; K = 6144 and 24576 take one either way)
        choose_splits(kblocks, count, dev->num_sms / 2, 24, &p.ksplit, &p.kb_per_split);
        p.tile_list = tiles;
        p.out = S;
        p.ldo = K;
        p.upper = 1;
        a.nprob = 1;
        // many waves of items (K = 24576: 4656 tiles, 62 waves): keep the pairs' waves
        // together (PairArgs::wave_ctr; measured 28.1-28.3 -> 25.1-27.5 ms for 65,536 tokens).
        // With 2-4 waves (K <= 6144) the pairs hardly drift apart and the waits cost about 1%.
        if (sched != nullptr && static_cast<int64_t>(count) * p.ksplit >= 16LL * (dev->num_sms / 2)) {
            a.wave_ctr = sched;
            a.exit_ctr = sched + 1;
        }
        a.status = dev->status;
        a.wait_limit_ns = wait_limit_ns();
        return launch_pair<true>(maps, a, dev, stream);
    }
    int count = 0;
    const int2* tiles = syrk_tiles(K, BM, 256, &count);
    if (tiles == nullptr) return cudaErrorMemoryAllocation;
    CUtensorMap mx, my;
    if (!encode_map(&mx, X, K, static_cast<uint64_t>(N), K, 64, BK)) return cudaErrorInvalidValue;
    if (!encode_map(&my, Y, K, static_cast<uint64_t>(N), K, 64, BK)) return cudaErrorInvalidValue;
    TcGemmArgs a{};
    a.rows = K;
    a.cols = K;
    a.kblocks = kblocks;
    a.tiles_n = 0;
    a.num_tiles = count;
    // this kernel accumulates a whole split in TMEM: splits of at most 1024 tokens keep the
    // fp32 accumulator precise (S is small whenever this path runs)
    a.kb_per_split = std::min(SYRK_CHUNK, kblocks);
    a.ksplit = (kblocks + a.kb_per_split - 1) / a.kb_per_split;
    a.tile_list = tiles;
    a.out = S;
    a.ldo = K;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    const int grid = std::min(a.num_tiles * a.ksplit, dev->num_sms);
    return launch_kernel<256, 4, true, EPI_ATOMIC_UPPER_F32>(mx, my, a, grid, stream);
}

cudaError_t launch_gemm_tn_tokens_f32(const void* U, int R, const void* V, int C, int64_t N, float* out,
                                     int64_t ldo, cudaStream_t stream)
{
    if (N <= 0 || R <= 0 || C <= 0) return cudaSuccess;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    if (dev->num_sms < 2) return cudaErrorInvalidConfiguration;
    CUtensorMap maps[4];
    if (!encode_map(&maps[0], U, R, static_cast<uint64_t>(N), R, 64, BK)) return cudaErrorInvalidValue;
    if (!encode_map(&maps[1], V, C, static_cast<uint64_t>(N), C, 64, BK)) return cudaErrorInvalidValue;
    maps[2] = maps[0];
    maps[3] = maps[1];
    PairArgs a{};
    PairProblem& p = a.p[0];
    p.rows = R;
    p.cols = C;
    p.kblocks = static_cast<int>((N + BK - 1) / BK);
    p.tiles_n = (C + PAIR_BN - 1) / PAIR_BN;
    p.num_tiles = ((R + PAIR_BM - 1) / PAIR_BM) * p.tiles_n;
    choose_splits(p.kblocks, p.num_tiles, dev->num_sms / 2, 8, &p.ksplit, &p.kb_per_split);
    p.tile_list = nullptr;
    p.out = out;
    p.ldo = ldo;
    p.upper = 0;
    a.nprob = 1;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_pair<true>(maps, a, dev, stream);
}

cudaError_t launch_gemm_nn(const void* A, int64_t lda, const void* B, int64_t ldb, int rows, int cols, int kdim,
                           void* C, int64_t ldc, cudaStream_t stream)
{
    if (rows <= 0 || cols <= 0) return cudaSuccess;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    if (dev->num_sms < 2) return cudaErrorInvalidConfiguration;
    CUtensorMap maps[4];
    if (!encode_map(&maps[0], A, kdim, rows, lda, BK, 128)) return cudaErrorInvalidValue;
    if (!encode_map(&maps[1], B, cols, kdim, ldb, 64, BK)) return cudaErrorInvalidValue;
    maps[2] = maps[0];
    maps[3] = maps[1];
    PairArgs a{};
    a.p[0] = pair_problem(rows, cols, kdim, C, ldc);
    a.nprob = 1;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_pair<false, true>(maps, a, dev, stream);
}

cudaError_t launch_forward_fused(const void* X, const void* PT, void* Z, const void* WfT, void* Y, int N,
                                 int K, int Lp, int M, int* ready, int* sched, cudaStream_t stream)
{
    if (N <= 0) return cudaSuccess;
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    if (dev->num_sms < 2) return cudaErrorInvalidConfiguration;
    CUtensorMap maps[4];
    if (!encode_map(&maps[0], X, K, N, K, BK, 128) || !encode_map(&maps[1], PT, K, Lp, K, BK, 128) ||
        !encode_map(&maps[2], Z, Lp, N, Lp, BK, 128) || !encode_map(&maps[3], WfT, Lp, M, Lp, BK, 128))
        return cudaErrorInvalidValue;
    PairArgs a{};
    a.p[0] = pair_problem(N, Lp, K, Z, Lp);
    a.p[1] = pair_problem(N, M, Lp, Y, M);
    a.nprob = 2;
    a.ready = ready;
    a.nready = (N + PAIR_BM - 1) / PAIR_BM;
    a.ticket = sched;
    a.exit_ctr = sched + 1;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_pair<false>(maps, a, dev, stream);
}

}  // namespace espace
