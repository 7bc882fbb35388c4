// decode.cu -- the projected forward for decode-shaped batches (N <= 32 tokens), HBM-bound.
//
// One cooperative launch computes both products of Eq. 3:
//   phase 1  Z[n][l] = bf16( sum_k X[n][k] P^T[l][k] )   P^T streamed from HBM once
//   -------  grid barrier -------------------------------------------------------------
//   phase 2  Y[n][m] = bf16( sum_l Z[n][l] W'^T[m][l] )  W'^T streamed once
// (and, with one phase only, the dense decode product Y = X W^T).
//
// Streaming. Each CTA owns a contiguous range of rows of each streamed matrix; the ranges
// are balanced over both phases together by bytes. One producer thread walks the CTA's
// stages -- (up to 8 rows) x (a k-block of up to SK elements) -- in the order they are
// consumed, phase 1 then phase 2, and copies each row piece into a ring of shared-memory
// stages with 1-D bulk copies (cp.async.bulk) completing on the stage's mbarrier. The
// producer does not wait for the grid barrier: while the consumers wait for Z, it keeps
// filling the ring with W'^T rows, so HBM stays busy across the barrier. (Holding the W'^T
// copies back until phase 1 has landed was measured slower: they then arrive as one burst
// just when the barrier's few L2 round trips are on the critical path.)
//
// Compute. The 16 consumer warps form groups of WPS warps (8 for N <= 8, 16 above); group q
// takes stages q, q + 16/WPS, .... For the dense product of one token, warp u of a group
// owns row u of each stage and runs fp32 FMA against the token, copied once to shared
// memory; otherwise the group's warps split the stage's k-block
// into 32-wide chunks. Each warp runs mma.sync.m16n8k16 (bf16 in, fp32 accumulate) with the
// tokens as the A operand (16 rows, rows >= N zero) and the 8 streamed rows as the B
// operand, one accumulator per chunk so consecutive MMAs do not wait on each other. The
// reduction index is permuted inside each 32-wide chunk: thread (g = lane / 4, t = lane % 4)
// reads elements 8t .. 8t+7 of streamed row g and of token rows g, g+8 with one 16-byte load
// each, which become k-slots {2t, 2t+1, 2t+8, 2t+9} of two consecutive k16 MMAs -- the same
// permutation on both operands, so the sum is unchanged. Stage rows sit at a pitch of
// SK * 2 + 16 bytes, so the 8 rows of one fragment load fall in different banks. A warp keeps
// its token fragments of the current k-block in registers. The WPS partial sums of a stage
// meet in a shared-memory fp32 accumulator (WPS-way atomic adds); each output is rounded to
// bf16 and written once.
//
// Grid barrier: each CTA adds to a counter whose bit 31 flips when all CTAs have arrived
// (one CTA adds 2^31 - (G - 1), the others 1; no reset between launches, the counter starts
// at zero). A CTA reads the bit when it starts -- it cannot flip before that CTA arrives --
// so arriving is one fire-and-forget release reduction, and waiting is acquire loads.
//
// Every wait is bounded: mbarrier waits, the producer's slot waits and the grid barrier give
// up after the wait limit, record ESPACE_ERR_TIMEOUT and leave; the producer then waits
// (bounded) for its copies in flight before the CTA exits.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "../../include/espace.h"
#include "kernels.h"
#include "ptx.cuh"

namespace espace {

constexpr int DEC_CWARPS = 16;                          // consumer warps
constexpr int DEC_THREADS = (DEC_CWARPS + 1) * 32;      // + one producer warp
constexpr int DEC_ROWS = 8;                             // streamed rows per stage
constexpr int DEC_MAX_STAGES = 12;
constexpr int DEC_MIN_STAGES = 4;
constexpr int DEC_SMEM_LIMIT = 232448;                  // opt-in shared memory per block, sm_103
constexpr int DEC_CONSUMER_BAR = 1;                     // named barrier of the consumer warps
constexpr int DEC_MAX_GRID = 192;                       // CTAs (one per SM) the cut tables hold

struct DecodeArgs {
    const __nv_bfloat16* A[2];   // streamed matrix of each phase, [R][kdim]
    const __nv_bfloat16* B[2];   // tokens of each phase, [nt][kdim]
    __nv_bfloat16* out[2];       // [nt][ldo]
    int R[2], kdim[2], ldo[2];
    int phases;                  // 1 (dense) or 2 (projected)
    int nt;
    int stages;                  // ring depth
    int acc_rows;                // rows of the shared accumulator
    int tok_elems;               // one token (N = 1): bf16 values of its shared-memory copy
    int slot_floats;             // 16-warp groups: floats of the partial-sum slots
    unsigned int* bar;           // grid barrier counter
    // launched with programmatic stream serialization: the producer streams the weights
    // (which the preceding grid must not write) before that grid has completed; the
    // consumers wait for it before reading tokens or touching the barrier counter
    int pdl;
    int* status;
    uint64_t wait_limit_ns;
    // CTA b owns rows [cut[p][b], cut[p][b + 1]) of phase p (computed on the host)
    int cut[2][DEC_MAX_GRID + 1];
};

// Row cuts: phase 1 split evenly over the G CTAs; phase 2 split so that the bytes of both
// phases together are balanced (when that keeps the ranges monotone), else evenly. n1, n2:
// rows; w1, w2: bytes per row (in any common unit). Host code: the kernel reads the tables.
void decode_cuts(int G, int phases, int n1, int w1, int n2, int w2, int* cut1, int* cut2)
{
    for (int b = 0; b <= G; ++b) cut1[b] = static_cast<int>(static_cast<int64_t>(n1) * b / G);
    if (phases < 2) {
        for (int b = 0; b <= G; ++b) cut2[b] = 0;
        return;
    }
    const int64_t tot = static_cast<int64_t>(n1) * w1 + static_cast<int64_t>(n2) * w2;
    const int64_t max1 = (static_cast<int64_t>(n1) + G - 1) / G;
    if (tot / G >= max1 * w1) {
        // cumulative phase-2 end after CTA c: the bytes target minus the phase-1 bytes so far;
        // nondecreasing in c because each CTA's target share covers its phase-1 rows
        cut2[0] = 0;
        for (int c = 0; c < G; ++c) {
            const int64_t t = tot * (c + 1) / G - static_cast<int64_t>(cut1[c + 1]) * w1;
            const int64_t e = t < 0 ? 0 : t / w2;
            cut2[c + 1] = static_cast<int>(std::min<int64_t>(e, n2));
        }
        cut2[G] = n2;
    } else {
        for (int b = 0; b <= G; ++b) cut2[b] = static_cast<int>(static_cast<int64_t>(n2) * b / G);
    }
}

__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                               uint32_t a3, uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ void consumer_sync()
{
    asm volatile("bar.sync %0, %1;" ::"n"(DEC_CONSUMER_BAR), "n"(DEC_CWARPS * 32) : "memory");
}

__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned* p)
{
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Grid barrier over all CTAs of a cooperative launch, by one thread per CTA; `start` is the
// counter as this thread read it when the CTA started. Every CTA arrives exactly once per
// launch, also one that has given up (skip_wait), so that the counter's bit flips once per
// launch and the next launch starts from a consistent count. Returns false (recording a
// timeout) if the others did not arrive within the limit, or at once with skip_wait.
__device__ bool grid_arrive_and_wait(unsigned* bar, unsigned start, int* status, uint64_t limit_ns, bool skip_wait)
{
    const unsigned nb = blockIdx.x == 0 ? 0x80000000u - (gridDim.x - 1) : 1u;
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(bar), "r"(nb) : "memory");
    if (skip_wait) return false;
    const uint64_t t0 = globaltimer_ns();
    uint32_t spins = 0;
    while (((start ^ ld_acquire_gpu(bar)) & 0x80000000u) == 0) {
        if ((++spins & 15u) == 0 && globaltimer_ns() - t0 > limit_ns) {
            atomicExch(status, ESPACE_ERR_TIMEOUT);
            return false;
        }
    }
    return true;
}

template <int MT, bool HI>
struct DecodeCfg {
    static constexpr int SK = 2048;                           // k-block of one stage
    // consumer warps per stage: each group of WPS warps takes every NG-th stage and splits its
    // k-block; wider token tiles use larger groups so the fragments fit the register budget
    static constexpr int WPS = (HI && MT > 0) ? 16 : 8;
    static constexpr int NG = DEC_CWARPS / WPS;
    static constexpr int CPW = SK / 32 / WPS;                 // 32-wide chunks per warp and stage
    static constexpr int NACC = MT == 2 ? 1 : CPW < 4 ? CPW : 4;   // independent MMA accumulators
    static constexpr int PITCH = SK * 2 + 16;                 // bytes per stage row
    static constexpr int STAGE_BYTES = DEC_ROWS * PITCH;
    // accumulator row pitch (floats): 16 tokens per m16 tile plus 4, so the lanes of one
    // flush (rows 2t, 2t+1; tokens g) hit 32 different banks
    static constexpr int NTP = MT == 0 ? 1 : 16 * MT + 4;
    // two token tiles (N > 16): a stage's partial sums meet through per-warp slots in shared
    // memory (double-buffered, [warp][8 rows][NTP]) instead of contended atomics (measured
    // faster there, slower for one tile)
    static constexpr bool SLOTS = MT == 2;
    static constexpr int SLOT_FLOATS = SLOTS ? 2 * 16 * DEC_ROWS * NTP : 0;
};

// A warp's token fragments for one k-block: v[chunk][m16 tile][row g / row g + 8].
template <int MT, bool HI>
struct TokFrag {
    uint4 v[DecodeCfg<MT, HI>::CPW][MT][HI ? 2 : 1];
};
// One token (MT = 0): lane l holds the token's fp32 values at k = 256 c + 8 l + e of the
// k-block, x[8 c + e].
template <>
struct TokFrag<0, false> {
    float x[64];
};

// Stage layout. When one k-block covers whole rows (kdim <= SK), a stage's rows are
// contiguous in HBM and arrive as two runs of 4 rows (two bulk copies), the second 64 bytes
// past the end of the first, so that the 8 rows of one fragment load still fall in different
// banks; otherwise each row piece is a copy of its own at a pitch of SK * 2 + 16 bytes.
template <int PITCH>
__device__ __forceinline__ int stage_row_offset(int row, int kdim, bool whole)
{
    return whole ? row * kdim * 2 + (row >= 4 ? 64 : 0) : row * PITCH;
}

template <int MT, bool HI>
__device__ __forceinline__ void load_tokens(TokFrag<MT, HI>& T, const __nv_bfloat16* B, bool coherent, int kdim,
                                            int nt, int kb, int u, int g, int t)
{
    using C = DecodeCfg<MT, HI>;
    if constexpr (MT == 0) {
        // B is the CTA's shared-memory copy of the token here
        const int lane = g * 4 + t;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
            const int k = kb * C::SK + 256 * c + 8 * lane;
            uint4 v = make_uint4(0, 0, 0, 0);
            if (k < kdim) v = *reinterpret_cast<const uint4*>(B + k);
            const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                T.x[8 * c + 2 * e] = __uint_as_float(w[e] << 16);
                T.x[8 * c + 2 * e + 1] = __uint_as_float(w[e] & 0xffff0000u);
            }
        }
        return;
    } else {
#pragma unroll
    for (int c = 0; c < C::CPW; ++c) {
        const int k = kb * C::SK + 32 * (u * C::CPW + c) + 8 * t;
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
            for (int h = 0; h < (HI ? 2 : 1); ++h) {
                const int n = mt * 16 + g + 8 * h;
                uint4 v = make_uint4(0, 0, 0, 0);
                if (n < nt && k < kdim) {
                    const uint4* p = reinterpret_cast<const uint4*>(B + static_cast<int64_t>(n) * kdim + k);
                    v = coherent ? __ldcg(p) : __ldg(p);
                }
                T.v[c][mt][h] = v;
            }
        }
    }
    }
}

// One stage for the warp with k-part u: the MMAs over its chunks, release of the stage, and
// the flush of its partial sums into acc (rows r0l .. r0l+rows-1 of the accumulator).
template <int MT, bool HI>
__device__ __forceinline__ void consume_stage(const unsigned char* st, uint64_t* empty_bar, const TokFrag<MT, HI>& T,
                                              int ksz, bool whole, int rows, int r0l, int nt, float* acc, int u,
                                              int lane, float* slot)
{
    using C = DecodeCfg<MT, HI>;
    if constexpr (MT == 0) {
        // one token: warp u owns row u of the stage and reads it 512 contiguous bytes at a
        // time; fp32 FMA into four accumulators, then one warp reduction per row
        float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
        if (u < rows) {
            const unsigned char* rp = st + stage_row_offset<C::PITCH>(u, ksz, whole);
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const int kl = 256 * c + 8 * lane;
                if (kl < ksz) {
                    const uint4 w = *reinterpret_cast<const uint4*>(rp + kl * 2);
                    s0 = fmaf(__uint_as_float(w.x << 16), T.x[8 * c + 0], s0);
                    s1 = fmaf(__uint_as_float(w.x & 0xffff0000u), T.x[8 * c + 1], s1);
                    s2 = fmaf(__uint_as_float(w.y << 16), T.x[8 * c + 2], s2);
                    s3 = fmaf(__uint_as_float(w.y & 0xffff0000u), T.x[8 * c + 3], s3);
                    s0 = fmaf(__uint_as_float(w.z << 16), T.x[8 * c + 4], s0);
                    s1 = fmaf(__uint_as_float(w.z & 0xffff0000u), T.x[8 * c + 5], s1);
                    s2 = fmaf(__uint_as_float(w.w << 16), T.x[8 * c + 6], s2);
                    s3 = fmaf(__uint_as_float(w.w & 0xffff0000u), T.x[8 * c + 7], s3);
                }
            }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(empty_bar);
        float sum = (s0 + s1) + (s2 + s3);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (lane == 0 && u < rows) atomicAdd(acc + (r0l + u) * C::NTP, sum);
        return;
    } else {
    const int g = lane >> 2, t = lane & 3;
    st += stage_row_offset<C::PITCH>(g, ksz, whole);
    float d[C::NACC][MT][4];
#pragma unroll
    for (int q = 0; q < C::NACC; ++q)
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) d[q][mt][0] = d[q][mt][1] = d[q][mt][2] = d[q][mt][3] = 0.f;
#pragma unroll
    for (int c = 0; c < C::CPW; ++c) {
        const int kl = 32 * (u * C::CPW + c) + 8 * t;
        uint4 w = make_uint4(0, 0, 0, 0);
        if (kl < ksz) w = *reinterpret_cast<const uint4*>(st + kl * 2);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
            const uint4 lo = T.v[c][mt][0];
            const uint4 hi = HI ? T.v[c][mt][HI ? 1 : 0] : make_uint4(0, 0, 0, 0);
            mma_bf16_16816(d[c % C::NACC][mt], lo.x, hi.x, lo.y, hi.y, w.x, w.y);
            mma_bf16_16816(d[c % C::NACC][mt], lo.z, hi.z, lo.w, hi.w, w.z, w.w);
        }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(empty_bar);
#pragma unroll
    for (int q = 1; q < C::NACC; ++q)
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int e = 0; e < 4; ++e) d[0][mt][e] += d[q][mt][e];
    // d[0][mt]: {token g, rows 2t, 2t+1}, {token g+8, rows 2t, 2t+1}
    if constexpr (C::SLOTS) {
        // this warp's slot; the rows and tokens that count are picked when the slots are summed
        float* sl = slot + (u * DEC_ROWS + 2 * t) * C::NTP;
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
            const int n = mt * 16 + g;
            sl[n] = d[0][mt][0];
            sl[C::NTP + n] = d[0][mt][1];
            sl[n + 8] = d[0][mt][2];
            sl[C::NTP + n + 8] = d[0][mt][3];
        }
        return;
    }
    // rows past the CTA's range were not copied and are not flushed
    const bool r_lo = 2 * t < rows, r_hi = 2 * t + 1 < rows;
    float* a = acc + (r0l + 2 * t) * C::NTP;
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
        const int n = mt * 16 + g;
        if (n < nt) {
            if (r_lo) atomicAdd(a + n, d[0][mt][0]);
            if (r_hi) atomicAdd(a + C::NTP + n, d[0][mt][1]);
        }
        if (HI && n + 8 < nt) {
            if (r_lo) atomicAdd(a + n + 8, d[0][mt][2]);
            if (r_hi) atomicAdd(a + C::NTP + n + 8, d[0][mt][3]);
        }
    }
    }
}

template <int MT, bool HI>
__global__ void __launch_bounds__(DEC_THREADS, 1) decode_kernel(const DecodeArgs a)
{
    using C = DecodeCfg<MT, HI>;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) uint64_t full[DEC_MAX_STAGES];
    __shared__ __align__(8) uint64_t empty[DEC_MAX_STAGES];
    __shared__ int abort_s;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int rb0[2] = {a.cut[0][blockIdx.x], a.cut[1][blockIdx.x]};   // rows [rb0[p], rb1[p])
    const int rb1[2] = {a.cut[0][blockIdx.x + 1], a.cut[1][blockIdx.x + 1]};


    float* acc = reinterpret_cast<float*>(smem);
    const size_t acc_bytes = (static_cast<size_t>(a.acc_rows) * C::NTP * 4 + 127) & ~static_cast<size_t>(127);
    __nv_bfloat16* tok_s = reinterpret_cast<__nv_bfloat16*>(smem + acc_bytes);
    const size_t tok_bytes = (static_cast<size_t>(a.tok_elems) * 2 + 127) & ~static_cast<size_t>(127);
    float* slots = reinterpret_cast<float*>(smem + acc_bytes + tok_bytes);
    unsigned char* ring = smem + acc_bytes + tok_bytes +
                          ((static_cast<size_t>(a.slot_floats) * 4 + 127) & ~static_cast<size_t>(127));

    if (threadIdx.x == 0) {
        for (int s = 0; s < a.stages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], C::WPS);
        }
        abort_s = 0;
        fence_barrier_init();
    }
    for (int i = threadIdx.x; i < a.acc_rows * C::NTP; i += blockDim.x) acc[i] = 0.f;
    __syncthreads();
    volatile int* abort = &abort_s;
    if (a.pdl && threadIdx.x == 0) grid_dep_launch_dependents();

    if (warp == DEC_CWARPS) {
        // ------------------------------------------------------------ producer (one thread)
        if (lane != 0) return;
        int j = 0;
#pragma unroll
        for (int p = 0; p < 2; ++p) {
            if (p >= a.phases || *abort) break;
            const __nv_bfloat16* A = a.A[p];
            const int kdim = a.kdim[p];
            const int nkb = (kdim + C::SK - 1) / C::SK;
            for (int kb = 0; kb < nkb && !*abort; ++kb) {
                const int ksz = min(C::SK, kdim - kb * C::SK);
                for (int r = rb0[p]; r < rb1[p]; r += DEC_ROWS, ++j) {
                    const int slot = j % a.stages;
                    if (j >= a.stages &&
                        !mbar_wait(&empty[slot], static_cast<uint32_t>(j / a.stages - 1) & 1u, abort, a.status,
                                   a.wait_limit_ns, ESPACE_ERR_TIMEOUT))
                        break;
                    const int rows = min(DEC_ROWS, rb1[p] - r);
                    mbar_arrive_expect_tx(&full[slot], static_cast<uint32_t>(rows * ksz * 2));
                    unsigned char* dst = ring + static_cast<size_t>(slot) * C::STAGE_BYTES;
                    const __nv_bfloat16* src = A + static_cast<int64_t>(r) * kdim + kb * C::SK;
                    if (kdim <= C::SK) {
                        // whole rows: two runs of up to 4 contiguous rows
                        const int lo = min(rows, 4);
                        bulk_load(dst, src, static_cast<uint32_t>(lo * kdim * 2), &full[slot]);
                        if (rows > 4)
                            bulk_load(dst + stage_row_offset<C::PITCH>(4, kdim, true), src + static_cast<int64_t>(4) * kdim,
                                      static_cast<uint32_t>((rows - 4) * kdim * 2), &full[slot]);
                    } else {
                        for (int q = 0; q < rows; ++q)
                            bulk_load(dst + q * C::PITCH, src + static_cast<int64_t>(q) * kdim,
                                      static_cast<uint32_t>(ksz * 2), &full[slot]);
                    }
                }
            }
        }
        if (*abort) {
            // let the copies already issued land before the CTA's shared memory goes away
            volatile int never = 0;
            for (int q = max(0, j - a.stages); q < j; ++q)
                mbar_wait(&full[q % a.stages], static_cast<uint32_t>(q / a.stages) & 1u, &never, a.status,
                          cleanup_limit(a.wait_limit_ns), ESPACE_ERR_TIMEOUT);
        }
        return;
    }

    // ---------------------------------------------------------------- consumers (16 warps)
    const int group = warp / C::WPS, u = warp % C::WPS;
    // tokens, Z and the barrier counter may belong to the preceding grid until it completes
    if (a.pdl) grid_dep_wait();
    // the grid barrier's bit before this CTA arrives (it cannot flip earlier)
    const unsigned bar_start = (a.phases > 1 && threadIdx.x == 0) ? ld_acquire_gpu(a.bar) : 0u;
    int j0 = 0;   // ring index of the phase's first stage
#pragma unroll
    for (int p = 0; p < 2; ++p) {
        if (p >= a.phases) break;
        const __nv_bfloat16* B = a.B[p];
        const bool coherent = p > 0;   // Z was written earlier in this launch
        const int kdim = a.kdim[p];
        const int nkb = (kdim + C::SK - 1) / C::SK;
        const int nrs = (rb1[p] - rb0[p] + DEC_ROWS - 1) / DEC_ROWS;   // row stages per k-block
        // stages run k-block-major; this group takes stages group, group + NG, ...
        if constexpr (MT == 0) {
            // one token: copy it to shared memory once (one 16-byte load per thread and
            // round), so that each warp reads it from there rather than from L2
            for (int k = 8 * threadIdx.x; k < kdim; k += 8 * DEC_CWARPS * 32) {
                const uint4* src = reinterpret_cast<const uint4*>(B + k);
                *reinterpret_cast<uint4*>(tok_s + k) = coherent ? __ldcg(src) : __ldg(src);
            }
            consumer_sync();
            B = tok_s;
        }
        TokFrag<MT, HI> T;
        int cur_kb = -1;
        for (int i = group; i < nkb * nrs; i += C::NG) {
            const int kb = i / nrs, rs = i - kb * nrs;
            if (kb != cur_kb) {
                load_tokens<MT, HI>(T, B, coherent, kdim, a.nt, kb, u, lane >> 2, lane & 3);
                cur_kb = kb;
            }
            const int j = j0 + i;
            const int slot = j % a.stages;
            const int r0l = rs * DEC_ROWS;
            const int srows = min(DEC_ROWS, rb1[p] - rb0[p] - r0l);
            float* slot_buf = slots + (i & 1) * (C::SLOT_FLOATS / 2);
            const bool ok = !*abort && mbar_wait(&full[slot], static_cast<uint32_t>(j / a.stages) & 1u, abort,
                                                 a.status, a.wait_limit_ns, ESPACE_ERR_TIMEOUT);
            if (ok)
                consume_stage<MT, HI>(ring + static_cast<size_t>(slot) * C::STAGE_BYTES, &empty[slot], T,
                                      min(C::SK, kdim - kb * C::SK), kdim <= C::SK, srows, r0l, a.nt, acc, u, lane,
                                      slot_buf);
            if constexpr (C::SLOTS) {
                // every consumer warp takes every stage (one group): one barrier per stage,
                // reached by all of them whatever happened above; then one thread per
                // (row, token) adds the 16 warps' slots in warp order (the double buffer lets
                // the next stage's slots be written before everyone has read these)
                consumer_sync();
                if (!*abort) {
                    const int e = threadIdx.x, r = e / C::NTP, n = e - r * C::NTP;
                    if (e < DEC_ROWS * C::NTP && r < srows && n < a.nt) {
                        float sum = 0.f;
#pragma unroll
                        for (int w = 0; w < DEC_CWARPS; ++w) sum += slot_buf[(w * DEC_ROWS + r) * C::NTP + n];
                        acc[(r0l + r) * C::NTP + n] += sum;
                    }
                }
            }
        }
        j0 += nkb * nrs;
        consumer_sync();
        // outputs of this CTA's rows, token-major (coalesced); then clear the accumulator
        const int rows = rb1[p] - rb0[p];
        if (!*abort) {
            for (int i = threadIdx.x; i < rows * a.nt; i += DEC_CWARPS * 32) {
                const int n = i / rows, rr = i - n * rows;
                a.out[p][static_cast<int64_t>(n) * a.ldo[p] + rb0[p] + rr] = __float2bfloat16_rn(acc[rr * C::NTP + n]);
            }
        }
        consumer_sync();
        for (int i = threadIdx.x; i < rows * C::NTP; i += DEC_CWARPS * 32) acc[i] = 0.f;
        if (p + 1 < a.phases) {
            // every Z of this CTA is stored (consumer_sync above); wait for all CTAs
            if (threadIdx.x == 0) {
                const bool ok = grid_arrive_and_wait(a.bar, bar_start, a.status, a.wait_limit_ns, *abort != 0);
                if (!ok) *abort = 1;
            }
        }
        consumer_sync();
    }
    if (threadIdx.x == 0 && *abort) {
        // copies the producer issued before the abort may still be landing in the ring
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 200000ull) __nanosleep(1000);
    }
}

// ------------------------------------------------------------------------------ host side

namespace {

struct DecodePlan {
    int mt = 1;
    bool hi = false;
    int stages = 0;
    int acc_rows = 0;
    int tok_elems = 0;
    int slot_floats = 0;
    int smem = 0;
    int cut[2][DEC_MAX_GRID + 1] = {};
};

int ntp_of(int mt) { return mt == 0 ? 1 : 16 * mt + 4; }
int stage_bytes_of(int) { return DecodeCfg<1, false>::STAGE_BYTES; }

bool compute_plan(int mt, bool hi, int phases, int R0, int k0, int R1, int k1, int G, DecodePlan* pl)
{
    pl->mt = mt;
    pl->hi = hi;
    decode_cuts(G, phases, R0, k0, phases > 1 ? R1 : 0, phases > 1 ? k1 : 1, pl->cut[0], pl->cut[1]);
    int max_rows = 1;
    for (int b = 0; b < G; ++b)
        max_rows = std::max(max_rows, std::max(pl->cut[0][b + 1] - pl->cut[0][b], pl->cut[1][b + 1] - pl->cut[1][b]));
    max_rows = (max_rows + DEC_ROWS - 1) / DEC_ROWS * DEC_ROWS;
    if (static_cast<int64_t>(max_rows) * ntp_of(mt) * 4 > DEC_SMEM_LIMIT) return false;
    pl->acc_rows = max_rows;
    const int acc_bytes = (pl->acc_rows * ntp_of(mt) * 4 + 127) & ~127;
    // one token: its shared-memory copy, for the longer of the two reductions
    pl->tok_elems = mt == 0 ? std::max(k0, phases > 1 ? k1 : 0) : 0;
    const int tok_bytes = (pl->tok_elems * 2 + 127) & ~127;
    pl->slot_floats = mt == 2 ? 2 * 16 * DEC_ROWS * ntp_of(mt) : 0;
    const int slot_bytes = (pl->slot_floats * 4 + 127) & ~127;
    const int sb = stage_bytes_of(mt);
    pl->stages = std::min(DEC_MAX_STAGES, (DEC_SMEM_LIMIT - 1024 - acc_bytes - tok_bytes - slot_bytes) / sb);
    if (pl->stages < DEC_MIN_STAGES) return false;
    pl->smem = acc_bytes + tok_bytes + slot_bytes + pl->stages * sb;
    return true;
}

// Plans are cached by shape: a decode step repeats the same few layer shapes.
bool make_plan(int nt, int phases, int R0, int k0, int R1, int k1, int G, DecodePlan* plan)
{
    if (nt < 1 || nt > DECODE_MAX_TOKENS || G < 1 || G > DEC_MAX_GRID) return false;
    if (k0 < 8 || k0 % 8 != 0 || R0 < 1) return false;
    if (phases > 1 && (k1 < 8 || k1 % 8 != 0 || R1 < 1)) return false;
    if (phases < 2) R1 = k1 = 0;
    // one token, one phase (the dense product): fp32 FMA with the token in shared memory; the
    // projected layer's two phases measured faster on the MMA path for one token too
    const int mt = (nt == 1 && phases == 1 && k0 <= 16384) ? 0 : nt <= 16 ? 1 : 2;
    const bool hi = mt > 0 && nt > 8;
    struct Entry {
        bool valid = false, ok = false;
        int key[8] = {};
        DecodePlan plan;
    };
    static Entry cache[16];
    static int next = 0;
    static std::mutex mu;
    const int key[8] = {mt, hi ? 1 : 0, phases, R0, k0, R1, k1, G};
    std::lock_guard<std::mutex> lock(mu);
    for (Entry& e : cache)
        if (e.valid && std::equal(key, key + 8, e.key)) {
            if (!e.ok) return false;
            *plan = e.plan;
            return true;
        }
    Entry& e = cache[next];
    next = (next + 1) % 16;
    e.valid = true;
    std::copy(key, key + 8, e.key);
    e.ok = compute_plan(mt, hi, phases, R0, k0, R1, k1, G, &e.plan);
    if (!e.ok) return false;
    *plan = e.plan;
    return true;
}

template <int MT, bool HI>
cudaError_t launch_t(DecodeArgs& a, const DecodePlan& pl, const DeviceInfo* dev, cudaStream_t stream)
{
    auto kern = decode_kernel<MT, HI>;
    static std::atomic<bool> configured[64];   // per device; a repeated set is harmless
    if (dev->device < 0 || dev->device >= 64) return cudaErrorInvalidDevice;
    if (!configured[dev->device].load(std::memory_order_acquire)) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             DEC_SMEM_LIMIT - 1024);
        if (e != cudaSuccess) return e;
        int per_sm = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, DEC_THREADS, DEC_SMEM_LIMIT - 1024);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) return cudaErrorInvalidConfiguration;
        configured[dev->device].store(true, std::memory_order_release);
    }
    a.stages = pl.stages;
    a.acc_rows = pl.acc_rows;
    a.tok_elems = pl.tok_elems;
    a.slot_floats = pl.slot_floats;
    std::copy(&pl.cut[0][0], &pl.cut[0][0] + 2 * (DEC_MAX_GRID + 1), &a.cut[0][0]);
    // programmatic stream serialization (see DecodeArgs::pdl), with a cooperative launch for
    // the grid barrier of the two-phase form
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(dev->num_sms);
    cfg.blockDim = dim3(DEC_THREADS);
    cfg.dynamicSmemBytes = static_cast<size_t>(pl.smem);
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    int na = 0;
    if (a.pdl) {
        attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    if (a.phases > 1) {
        attr[na].id = cudaLaunchAttributeCooperative;
        attr[na].val.cooperative = 1;
        ++na;
    }
    cfg.attrs = attr;
    cfg.numAttrs = na;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

cudaError_t launch_any(DecodeArgs& a, const DecodePlan& pl, const DeviceInfo* dev, cudaStream_t stream)
{
    if (pl.mt == 0) return launch_t<0, false>(a, pl, dev, stream);
    if (pl.mt == 2) return launch_t<2, true>(a, pl, dev, stream);
    if (pl.hi) return launch_t<1, true>(a, pl, dev, stream);
    return launch_t<1, false>(a, pl, dev, stream);
}

}  // namespace

bool decode_supported(int nt, int K, int Lp, int M, int num_sms)
{
    DecodePlan pl;
    return make_plan(nt, 2, Lp, K, M, Lp, num_sms, &pl);
}

bool decode_dense_supported(int nt, int K, int M, int num_sms)
{
    DecodePlan pl;
    return make_plan(nt, 1, M, K, 0, 0, num_sms, &pl);
}

cudaError_t launch_decode_forward(const void* PT, const void* WfT, const void* X, void* Z, void* Y,
                                  int K, int Lp, int M, int nt, unsigned int* grid_bar,
                                  cudaStream_t stream)
{
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    DecodePlan pl;
    if (!make_plan(nt, 2, Lp, K, M, Lp, dev->num_sms, &pl)) return cudaErrorInvalidValue;
    DecodeArgs a{};
    a.A[0] = static_cast<const __nv_bfloat16*>(PT);
    a.B[0] = static_cast<const __nv_bfloat16*>(X);
    a.out[0] = static_cast<__nv_bfloat16*>(Z);
    a.R[0] = Lp;
    a.kdim[0] = K;
    a.ldo[0] = Lp;
    a.A[1] = static_cast<const __nv_bfloat16*>(WfT);
    a.B[1] = static_cast<const __nv_bfloat16*>(Z);
    a.out[1] = static_cast<__nv_bfloat16*>(Y);
    a.R[1] = M;
    a.kdim[1] = Lp;
    a.ldo[1] = M;
    a.phases = 2;
    a.nt = nt;
    a.bar = grid_bar;
    a.pdl = 1;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_any(a, pl, dev, stream);
}

cudaError_t launch_decode_dense(const void* W, const void* X, void* Y, int K, int M, int nt,
                                cudaStream_t stream)
{
    DeviceInfo* dev = nullptr;
    if (device_info(&dev) != ESPACE_OK) return cudaErrorUnknown;
    DecodePlan pl;
    if (!make_plan(nt, 1, M, K, 0, 0, dev->num_sms, &pl)) return cudaErrorInvalidValue;
    DecodeArgs a{};
    a.A[0] = static_cast<const __nv_bfloat16*>(W);
    a.B[0] = static_cast<const __nv_bfloat16*>(X);
    a.out[0] = static_cast<__nv_bfloat16*>(Y);
    a.R[0] = M;
    a.kdim[0] = K;
    a.ldo[0] = M;
    a.phases = 1;
    a.nt = nt;
    a.bar = nullptr;
    a.pdl = 1;
    a.status = dev->status;
    a.wait_limit_ns = wait_limit_ns();
    return launch_any(a, pl, dev, stream);
}

}  // namespace espace
