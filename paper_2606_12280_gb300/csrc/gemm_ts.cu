// gemm_ts.cu -- the W8A8 linear (a4 + a5, dual-branch a6) on pairs of SMs with
// the weights in tensor memory: tcgen05.mma.cta_group::2 in its "TS" form
// (A operand in TMEM, B operand in shared memory).
//
// Same exact-integer scheme as gemm_tc2.cu: int8 values are fp16 values,
// products are exact in fp32, and partial sums of at most 1024 products stay
// below 2^24, so K advances in chunks of 1024 that are drained from TMEM into
// int32 running sums.  What changes is where each operand lives.  The
// activation codes arrive as fp16 values (the fp16-code variant of a3 writes
// them), so TMA puts them straight into the 128-byte swizzled B operand; the
// int8 weights are the A operand: TMA stages them in an int8 ring, the
// converter warps turn each CTA's 128 weight rows into fp16 in registers and
// write them into TMEM with tcgen05.st, and the MMA reads A from there.  Per SM
// and K=128 stage, shared memory then carries 16 KB of int8 weights (one TMA
// write, one converter read) and 32 KB of activations (one TMA write, one
// tensor-core read): no fp16 store of a converted operand and no tensor-core
// read of one.
//
// A cluster of two CTAs computes a 256 (output features) x 256 (tokens) tile
// of Y^T: CTA r holds weight rows f0 + 128r .. +127 in its TMEM lanes and the
// tokens t0 + 128r .. +127 in its shared memory; the leader issues M=256 N=256
// K=16 MMAs (eight per stage: N=256 keeps each instruction long enough for one
// issuing thread to keep the tensor pipe fed) and each CTA's TMEM receives its
// 128 feature rows x 256 tokens of the fp32 accumulator.  TMEM per CTA: one
// 256-column accumulator + four 64-column weight slots of K=128 = 512 columns.
// With a single accumulator the MMA waits at every K chunk until the
// epilogue has drained it; the drain is short (TMEM -> registers) and the
// stores of a finished tile overlap the next tile's first chunk.
//
// Per CTA: warp 0 TMA producer of the int8 weight ring, warp 2 TMA producer of
// the fp16 activation ring (both CTAs load against the leader's barrier, so
// the leader learns directly that both halves of B have landed), warp 1 TMEM
// allocation (both CTAs) and MMA issue (leader only), warps 4-7 converters
// (warp w owns TMEM lanes 32(w%4) .. +31, one weight row per thread), warps
// 8-15 epilogue (TMEM -> int32 running sums -> bf16 dequantized output, one
// output feature per thread).  Cross-CTA signalling: converters and epilogue
// warps arrive on the leader's barriers through cluster addresses; the leader
// commits MMA completion to both CTAs' barriers by multicast.  All waits are
// bounded in time.
#include <cstdint>
#include <type_traits>
#include <cuda.h>
#include <cuda_runtime.h>

#include "common.cuh"
#include "host_once.h"
#include "launch.h"
#include "tc_ptx.cuh"
#include "tile_order.cuh"

namespace w8a8 {
namespace {

using namespace tc;

#ifndef W8A8_TS_S8
#define W8A8_TS_S8 4
#endif
constexpr int PAIR_F = 256, CTA_F = 128;             // output features per pair / CTA (MMA M)
constexpr int PAIR_T = 256, CTA_T = 128;             // tokens per pair / CTA (MMA N)
constexpr int BK = 64;                               // K per sub-block (one swizzle atom row)
constexpr int SUB = 2;                               // sub-blocks per stage
constexpr int KC_BLOCKS = 16;                        // K chunk = 1024 (exactness bound)
static_assert(KC_BLOCKS * BK * 127 * 127 < (1 << 24), "fp32 exactness bound");
static_assert(KC_BLOCKS % SUB == 0, "chunk of whole stages");
constexpr int KC_STAGES = KC_BLOCKS / SUB;
// One slot index for the stage's weights in TMEM and its activations in
// shared memory, so that one barrier says "both landed" and one MMA commit
// frees both.
constexpr int SA = 4;                                // slots: TMEM weights + smem activations
constexpr int SX = SA;
constexpr int S8 = W8A8_TS_S8;                       // weight ring (int8, smem)
constexpr int SUBX = CTA_T * BK * 2;                 // 16 KB: one sub-block of activations
constexpr int SUBW = CTA_F * BK;                     // 8 KB: one sub-block of weights
constexpr int STAGE_X = SUB * SUBX;
constexpr int STAGE_W = SUB * SUBW;
constexpr uint32_t ACC_COLS = PAIR_T;                // fp32 columns of the accumulator
constexpr uint32_t A_COL0 = ACC_COLS;                // first weight-slot column
constexpr uint32_t A_SLOT_COLS = SUB * BK / 2;       // fp16 pairs per row of a slot
constexpr int TMEM_COLS = 512;
static_assert(A_COL0 + SA * A_SLOT_COLS <= TMEM_COLS, "tensor memory");
constexpr int NUM_CONV_WARPS = 4;
constexpr int NUM_EPI_WARPS = 8;
constexpr int THREADS = 512;
constexpr int LAUNCH_REGS = 128;
constexpr int REGS_LOW = 72, REGS_HIGH = 184;
static_assert(256 * REGS_LOW + 256 * REGS_HIGH <= THREADS * LAUNCH_REGS, "register split");
constexpr int RUN = PAIR_T / 2;                      // running sums per epilogue thread

constexpr unsigned ERR_PRODUCER = 1u, ERR_CONVERTER = 2u, ERR_MMA = 4u, ERR_EPILOGUE = 8u,
                   ERR_DRAIN = 16u, ERR_TMEM_PAIR = 64u;

constexpr uint32_t OFF_X = 0;
constexpr uint32_t OFF_W = OFF_X + SX * STAGE_X;
constexpr uint32_t OFF_BAR = OFF_W + S8 * STAGE_W;
constexpr uint32_t BAR_FULL8 = OFF_BAR;                     // weight stage landed (tx)
constexpr uint32_t BAR_EMPTY8 = BAR_FULL8 + 8 * S8;          // converters read it
// leader's: this slot's weights written by all converter warps of both CTAs
// (arrivals) and both CTAs' activations landed (transaction bytes, armed by
// the leader's activation producer, which also counts as one arrival)
constexpr uint32_t BAR_SFULL = BAR_EMPTY8 + 8 * S8;
constexpr uint32_t BAR_SEMPTY = BAR_SFULL + 8 * SA;          // MMA done with the slot (commit)
constexpr uint32_t BAR_ACCFULL = BAR_SEMPTY + 8 * SA;        // chunk accumulated
constexpr uint32_t BAR_ACCEMPTY = BAR_ACCFULL + 8;           // leader: chunk drained
constexpr uint32_t BAR_DRAIN = BAR_ACCEMPTY + 8;
constexpr uint32_t BAR_TFLAG = BAR_DRAIN + 8;              // a tile's single-run flag published
constexpr uint32_t OFF_TFLAG = BAR_TFLAG + 16;             // the flags (two tiles in flight)
constexpr uint32_t OFF_TMEM = OFF_TFLAG + 8;
constexpr uint32_t OFF_ABORT = OFF_TMEM + 4;
constexpr uint32_t OFF_SPLIT = OFF_ABORT + 4;                // a split part's arrival order
constexpr uint32_t SMEM_BARRIERS = 512;
static_assert(OFF_SPLIT + 4 - OFF_BAR <= SMEM_BARRIERS, "barrier area");
// per epilogue warp: the activation scales of its 128 tokens
constexpr uint32_t OFF_EPI = OFF_BAR + SMEM_BARRIERS;
constexpr uint32_t EPI_BYTES = (PAIR_T / 2) * 4;
constexpr int SMEM_TOTAL = 1024 + OFF_EPI + NUM_EPI_WARPS * EPI_BYTES;
static_assert(SMEM_TOTAL <= 232448, "shared memory");
static_assert(SUBX % 1024 == 0 && SUBW % 1024 == 0, "swizzle atoms stay aligned");

struct BranchArgs {
    const float *x_scale;
    const float *w_scale;
    const float *bias;
    void *out;
    const uint32_t *x_sumsq;   // per token sum of squared codes, or null
    const uint32_t *plan;      // the weights' drain plan (see plan_drains), or null
    int M;           // tokens
    int t_tiles;     // token tiles of 256
    int tiles;       // t_tiles * feature tiles
};

struct Params {
    BranchArgs br[2];
    int N, K;
    int total_tiles;
    int k_blocks;
    // per 256-row weight block of a branch's plan: plan_words words, the
    // drain bits (bit c set = drain after K chunk c), then the block's max
    // sum of squares
    int plan_words;
    // every branch has a plan and x_sumsq: tiles whose activation and weight
    // norms bound every partial sum run without an intermediate drain
    int single_ok;
    unsigned int *err;
    uint64_t wait_limit_ns;
    // work units: first the split_tiles last tiles as `split` parts each
    // over consecutive K chunks (split = 1: none), then tiles 0 ..
    // full_tiles - 1 whole; a part's int32 sums go to ws, and the last part
    // of a tile to arrive (ws_cnt) adds them up and runs the epilogue
    int full_tiles, split, split_tiles, total_units;
    // tile order: groups of group_f feature blocks; within a group the
    // feature block changes fastest (group_f = 1: the token tile changes
    // fastest, every feature block's tiles in a row)
    int f_tiles, group_f;
    int32_t *ws;               // [split_tiles][split][PAIR_T tokens][PAIR_F features]
    unsigned int *ws_cnt;      // [split_tiles][2 CTAs], zero between calls
};

struct Tile {
    int branch, t0, f0;
};

// Tile t of the launch's tile space: token tiles fastest, or (GROUPED) in
// groups of feature blocks as tile_order.cuh describes.  The plain order is
// its own instantiation: the benchmarked shapes use it, and a kernel whose
// tile loop carried the grouped arithmetic measured ~1 % slower on them.
template <bool GROUPED>
__device__ __forceinline__ Tile tile_coords(const Params &p, int t) {
    Tile r;
    r.branch = t >= p.br[0].tiles ? 1 : 0;
    const int local = t - (r.branch ? p.br[0].tiles : 0);
    const int tt = p.br[r.branch].t_tiles;
    if (GROUPED) {
        int ti, fi;
        grouped_tile(local, tt, p.f_tiles, p.group_f, ti, fi);
        r.t0 = ti * PAIR_T;
        r.f0 = fi * PAIR_F;
    } else {
        r.t0 = (local % tt) * PAIR_T;
        r.f0 = (local / tt) * PAIR_F;
    }
    return r;
}

struct Unit {
    int tile;          // output tile
    int ci0, ci1;      // K chunks [ci0, ci1)
    int part, slot;    // split part, split tile index (-1: a whole tile)
};

// The split parts come first, in the pairs' first round: the exchange of
// partial sums then overlaps the whole tiles that follow instead of
// lengthening the end of the kernel.
__device__ __forceinline__ Unit unit_coords(const Params &p, int u, int NC) {
    Unit r;
    const int nsplit = p.split_tiles * p.split;
    if (u >= nsplit) {
        r.tile = u - nsplit;
        r.ci0 = 0;
        r.ci1 = NC;
        r.part = 0;
        r.slot = -1;
    } else {
        r.slot = u / p.split;
        r.part = u - r.slot * p.split;
        r.tile = p.full_tiles + r.slot;
        r.ci0 = r.part * NC / p.split;
        r.ci1 = (r.part + 1) * NC / p.split;
    }
    return r;
}

// int8 x4 -> two fp16x2 words, exact (bytes + 128 in the mantissa of 1024.0,
// minus 1152).
// Does the accumulation stop (the epilogue drains TMEM) after K chunk ci of a
// tile of weight block fb?  Always after the tile's last chunk.
__device__ __forceinline__ bool plan_drains(const Params &p, const uint32_t *plan, int fb, int ci, int NC) {
    if (ci == NC - 1 || plan == nullptr) return true;
    return (__ldg(plan + (size_t)fb * p.plan_words + (ci >> 5)) >> (ci & 31)) & 1u;
}

// Can tile t run without an intermediate drain?  Every partial sum P over a
// subset S of K obeys |P| <= ||a_S|| ||w_S|| <= ||a|| ||w|| (Cauchy-Schwarz),
// so max_t ||a_t||^2 * max_f ||w_f||^2 <= 2^48 over the tile's 256 tokens and
// 256 weight rows keeps every one within 2^24, exact in fp32.  Warp-wide: all
// lanes take part.
template <bool GROUPED>
__device__ __forceinline__ bool tile_single_run(const Params &p, int t, int lane) {
    const Tile tl = tile_coords<GROUPED>(p, t);
    const BranchArgs &br = p.br[tl.branch];
    uint32_t m = 0;
#pragma unroll
    for (int i = lane; i < PAIR_T; i += 32)
        if (tl.t0 + i < br.M) m = max(m, __ldg(br.x_sumsq + tl.t0 + i));
    m = __reduce_max_sync(0xffffffffu, m);
    const uint32_t wm = __ldg(br.plan + (size_t)(tl.f0 / PAIR_F) * p.plan_words + p.plan_words - 1);
    return static_cast<uint64_t>(m) * wm <= (1ull << 48);
}

__device__ __forceinline__ void i8x4_to_f16x4(uint32_t w, uint32_t &lo, uint32_t &hi) {
    const uint32_t u = w ^ 0x80808080u;
    asm("prmt.b32 %0, %1, %2, 0x4140;" : "=r"(lo) : "r"(u), "r"(0x64646464u));
    asm("prmt.b32 %0, %1, %2, 0x4342;" : "=r"(hi) : "r"(u), "r"(0x64646464u));
    asm("sub.f16x2 %0, %0, %1;" : "+r"(lo) : "r"(0x64806480u));
    asm("sub.f16x2 %0, %0, %1;" : "+r"(hi) : "r"(0x64806480u));
}

// The int32 value of an fp32 integer v, |v| <= 2^24, without a conversion
// instruction (those run at a fraction of the add rate, and the MMA waits for
// the drain): t = v + 1.5 * 2^25 lies in [2^25, 2^26], where fp32 values are
// 4 apart, so t's bit pattern counts v rounded to a multiple of 4, t - 1.5 *
// 2^25 is that multiple exactly, and the rest (|lo| <= 2, exact) is read in
// the low mantissa bits of lo + 1.5 * 2^23.  The bit count stays linear at
// t = 2^26 (the mantissa carries into the exponent).
__device__ __forceinline__ int32_t exact_int(uint32_t vb) {
    const float v = __uint_as_float(vb);
    const float t = __fadd_rn(v, 50331648.0f);
    const float lo = __fadd_rn(v, -__fadd_rn(t, -50331648.0f));
    const uint32_t hi4 = (__float_as_uint(t) - 0x4C400000u) << 2;
    return static_cast<int32_t>(hi4 + (__float_as_uint(__fadd_rn(lo, 12582912.0f)) - 0x4B400000u));
}

// exact_int of two values at once with packed fp32 adds (same steps).
__device__ __forceinline__ void exact_int2(uint32_t v0, uint32_t v1, int32_t &r0, int32_t &r1) {
    uint64_t v, t, h, lo, m;
    asm("mov.b64 %0, {%1, %2};" : "=l"(v) : "r"(v0), "r"(v1));
    const uint64_t C = 0x4C4000004C400000ull, NC = 0xCC400000CC400000ull, M = 0x4B4000004B400000ull,
                   NEG1 = 0xBF800000BF800000ull;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(t) : "l"(v), "l"(C));
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(h) : "l"(t), "l"(NC));
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(lo) : "l"(h), "l"(NEG1), "l"(v));
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(m) : "l"(lo), "l"(M));
    uint32_t t0, t1, m0, m1;
    asm("mov.b64 {%0, %1}, %2;" : "=r"(t0), "=r"(t1) : "l"(t));
    asm("mov.b64 {%0, %1}, %2;" : "=r"(m0), "=r"(m1) : "l"(m));
    r0 = static_cast<int32_t>(((t0 - 0x4C400000u) << 2) + (m0 - 0x4B400000u));
    r1 = static_cast<int32_t>(((t1 - 0x4C400000u) << 2) + (m1 - 0x4B400000u));
}

__device__ __forceinline__ void arrive_leader(uint32_t bar, uint32_t rank) {
    if (rank == 0) mbar_arrive(bar);
    else mbar_arrive_cluster_relaxed(mapa_shared(bar, 0));
}

template <bool OUT_I32, bool GROUPED>
__device__ __forceinline__ void epilogue_role(const Params &p, uint32_t sb, uint32_t tmem,
                                              const WaitCtx &wc, int warp, int lane, int NC,
                                              uint32_t rank, int pair, int npairs) {
    const int q = warp & 3;            // TMEM lane quarter this warp may access
    const int h = (warp - 8) >> 2;     // token half of the 256-wide tile
    uint32_t c = 0;                    // drains so far
    bool ok = true;
    // single-run tiles: every warp decides for itself (the same inputs give
    // the same answer in both CTAs); warp 8 of the leader publishes the
    // answer for the MMA thread, one tile ahead, so it never waits for it
    const bool use_single = p.single_ok != 0;
    const bool publisher = use_single && rank == 0 && warp == 8;
    auto publish = [&](int n, bool v) {
        if (publisher && lane == 0) {
            st_shared_s32(sb + OFF_TFLAG + 4 * (n & 1), v ? 1 : 0);
            mbar_arrive(sb + BAR_TFLAG + 8 * (n & 1));
        }
    };
    bool single = use_single && pair < p.total_units && tile_single_run<GROUPED>(p, unit_coords(p, pair, NC).tile, lane);
    if (pair < p.total_units) publish(0, single);
    int n = 0;                         // units so far
    for (int u = pair; ok && u < p.total_units; u += npairs, ++n) {
        const Unit un = unit_coords(p, u, NC);
        const int t = un.tile;
        const Tile tc = tile_coords<GROUPED>(p, t);
        const int fb = tc.f0 / PAIR_F;
        const uint32_t *plan = p.br[tc.branch].plan;
        int32_t run[RUN];
#pragma unroll
        for (int i = 0; i < RUN; ++i) run[i] = 0;
        for (int ci = un.ci0; ci < un.ci1; ++ci) {
            if (ci != un.ci1 - 1 && (single || !plan_drains(p, plan, fb, ci, NC))) continue;
            if (!mbar_wait_cluster(sb + BAR_ACCFULL, c & 1, wc, ERR_EPILOGUE)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t base = tmem + (static_cast<uint32_t>(q * 32) << 16) + h * (PAIR_T / 2);
            // two loads in flight per wait: the MMA is stopped until every
            // epilogue warp has drained its part.  A tile's only run is kept
            // as fp32 (its values are the exact integers, and (float)acc is
            // all the epilogue needs); otherwise the values are read with
            // adds instead of conversion instructions (exact_int)
            if (single) {
#pragma unroll
                for (int jj = 0; jj < RUN / 16; jj += 4) {
                    uint32_t v[4][16];
#pragma unroll
                    for (int g = 0; g < 4; ++g) tmem_ld_32x32b_x16(base + (jj + g) * 16, v[g]);
                    tmem_ld_wait();
#pragma unroll
                    for (int g = 0; g < 4; ++g)
#pragma unroll
                        for (int i = 0; i < 16; ++i) run[(jj + g) * 16 + i] = static_cast<int32_t>(v[g][i]);
                }
            } else {
#pragma unroll
                for (int jj = 0; jj < RUN / 16; jj += 2) {
                    uint32_t v[2][16];
#pragma unroll
                    for (int g = 0; g < 2; ++g) tmem_ld_32x32b_x16(base + (jj + g) * 16, v[g]);
                    tmem_ld_wait();
#pragma unroll
                    for (int g = 0; g < 2; ++g)
#pragma unroll
                        for (int i = 0; i < 16; i += 2) {
                            int32_t r0, r1;
                            exact_int2(v[g][i], v[g][i + 1], r0, r1);
                            run[(jj + g) * 16 + i] += r0;
                            run[(jj + g) * 16 + i + 1] += r1;
                        }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) arrive_leader(sb + BAR_ACCEMPTY, rank);
            ++c;
        }
        if (!ok) break;
        // the next unit's decision, before this unit's stores
        bool raw = single;
        if (use_single) {
            const int un_next = u + npairs;
            single = un_next < p.total_units && tile_single_run<GROUPED>(p, unit_coords(p, un_next, NC).tile, lane);
            if (un_next < p.total_units) publish(n + 1, single);
        }
        if (un.slot >= 0) {
            // a part of a split tile: this warp's 32 features x 128 tokens of
            // int32 sums go to the workspace, and the warp of the part that
            // arrives last adds the other parts' and stores the tile (integer
            // sums: exact in any order).  Each warp counts its own arrivals,
            // so no warp waits for another.
            if (raw) {
#pragma unroll
                for (int i = 0; i < RUN; ++i) run[i] = exact_int(static_cast<uint32_t>(run[i]));
                raw = false;
            }
            const size_t at = (size_t)h * (PAIR_T / 2) * PAIR_F + rank * CTA_F + q * 32 + lane;
            const size_t part_elems = (size_t)PAIR_T * PAIR_F;
            int32_t *mine = p.ws + (size_t)(un.slot * p.split + un.part) * part_elems + at;
#pragma unroll
            for (int i = 0; i < RUN; ++i) __stcg(mine + (size_t)i * PAIR_F, run[i]);
            __threadfence();
            __syncwarp();
            unsigned int *cnt = p.ws_cnt + (size_t)un.slot * 16 + rank * 8 + (warp - 8);
            unsigned int order = 0;
            if (lane == 0) order = atomicAdd(cnt, 1u);
            order = __shfl_sync(0xffffffffu, order, 0);
            if (order != static_cast<unsigned int>(p.split - 1)) {
                __syncwarp();
                continue;
            }
            __threadfence();
            for (int pp = 0; pp < p.split; ++pp) {
                if (pp == un.part) continue;
                const int32_t *other = p.ws + (size_t)(un.slot * p.split + pp) * part_elems + at;
                // 32 loads in flight per batch
#pragma unroll
                for (int jb = 0; jb < RUN; jb += 32) {
                    int32_t tmp[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) tmp[i] = __ldcg(other + (size_t)(jb + i) * PAIR_F);
#pragma unroll
                    for (int i = 0; i < 32; ++i) run[jb + i] += tmp[i];
                }
            }
            if (lane == 0) *cnt = 0u;          // every part has arrived: ready for the next call
        }
        // one representation for the stores: int32 for the int32 export,
        // fp32 (the exact value, |acc| <= 2^24 or rounded as (float)acc)
        // for the dequantized output
#pragma unroll
        for (int i = 0; i < RUN; ++i) {
            if (OUT_I32) {
                if (raw) run[i] = exact_int(static_cast<uint32_t>(run[i]));
            } else if (!raw) {
                run[i] = static_cast<int32_t>(__float_as_uint(__int2float_rn(run[i])));
            }
        }
        const Tile tl = tile_coords<GROUPED>(p, t);
        const BranchArgs &br = p.br[tl.branch];
        const int f = tl.f0 + static_cast<int>(rank) * CTA_F + q * 32 + lane;   // output feature
        const int tok0 = tl.t0 + h * (PAIR_T / 2);
        const int ntok = min(RUN, br.M - tok0);
        const bool fok = f < p.N;
        if (ntok > 0) {             // uniform across the warp (one token range)
            if (OUT_I32 && fok) {
                int32_t *out = static_cast<int32_t *>(br.out) + (size_t)tok0 * p.N + f;
#pragma unroll
                for (int i = 0; i < RUN; ++i)
                    if (i < ntok) out[(size_t)i * p.N] = run[i];
            } else if (!OUT_I32) {
                const float sw = fok ? __ldg(br.w_scale + f) : 0.0f;
                const bool hb = br.bias != nullptr;
                const float b = (hb && fok) ? __ldg(br.bias + f) : 0.0f;
                // the warp's 128 token scales go through shared memory once
                // (one 16-byte load per lane), then every lane reads them as
                // broadcasts: a global load per token inside the store loop
                // would wait a full memory latency per token
                const uint32_t epi = sb + OFF_EPI + (warp - 8) * EPI_BYTES;
                bool sx_ok;
                {
                    const float *sxp = br.x_scale + tok0;
                    float4 s4;
                    if (4 * lane + 3 < ntok) {
                        s4 = __ldg(reinterpret_cast<const float4 *>(sxp) + lane);
                    } else {
                        s4.x = 4 * lane < ntok ? __ldg(sxp + 4 * lane) : 0.0f;
                        s4.y = 4 * lane + 1 < ntok ? __ldg(sxp + 4 * lane + 1) : 0.0f;
                        s4.z = 4 * lane + 2 < ntok ? __ldg(sxp + 4 * lane + 2) : 0.0f;
                        s4.w = 0.0f;
                    }
                    st_shared_v4(epi + 16 * lane, make_uint4(__float_as_uint(s4.x), __float_as_uint(s4.y),
                                                             __float_as_uint(s4.z), __float_as_uint(s4.w)));
                    constexpr float kSxLimit = 0x1p96f;       // |acc| < 2^31: acc * sx stays finite
                    sx_ok = fabsf(s4.x) <= kSxLimit && fabsf(s4.y) <= kSxLimit && fabsf(s4.z) <= kSxLimit &&
                            fabsf(s4.w) <= kSxLimit;
                    __syncwarp();
                }
                // lanes 2i and 2i+1 (features f, f+1) swap one value per pair
                // of tokens, so that each stores one 32-bit word: the even
                // lane both features of the first token, the odd lane both of
                // the second (N is a multiple of 8, so the word is 4-byte
                // aligned and both features of a pair are inside).  No output
                // of the tile can be a NaN when every scale and the bias are
                // finite and |sx| <= 2^96: acc * sx is then finite, times sw
                // it may overflow to an infinity, and a finite bias leaves
                // that infinite.  Each pair is then rounded to bf16 by one
                // conversion instruction.  The epilogue shares the SM's issue
                // slots with the converters, and rounding every value with
                // integer operations made the whole GEMM ~5 % slower; tiles
                // that could hold a NaN keep that rounding, which preserves a
                // NaN's payload.
                const bool odd = lane & 1;
                const int fw = f & ~1;
                uint16_t *out = static_cast<uint16_t *>(br.out) + (size_t)tok0 * p.N + fw;
                const bool fast_cvt = __all_sync(0xffffffffu, sx_ok && fabsf(sw) <= 3.402823466e38f &&
                                                                   (!hb || fabsf(b) <= 3.402823466e38f));
                auto store_pairs = [&](auto fast_tag) {
                    constexpr bool FAST = decltype(fast_tag)::value;
#pragma unroll
                    for (int i = 0; i < RUN; i += 4) {
                        const uint4 s4 = ld_shared_v4(epi + 4 * i);
                        const float sxv[4] = {__uint_as_float(s4.x), __uint_as_float(s4.y), __uint_as_float(s4.z),
                                              __uint_as_float(s4.w)};
#pragma unroll
                        for (int u = 0; u < 4; u += 2) {
                            const float t0 = epilogue_f32(__uint_as_float(static_cast<uint32_t>(run[i + u])),
                                                          sxv[u], sw, b, hb);
                            const float t1 = epilogue_f32(__uint_as_float(static_cast<uint32_t>(run[i + u + 1])),
                                                          sxv[u + 1], sw, b, hb);
                            const float other = __shfl_xor_sync(0xffffffffu, odd ? t0 : t1, 1);
                            const int tk = i + u + (odd ? 1 : 0);
                            const float lo = odd ? other : t0, hi = odd ? t1 : other;
                            const uint32_t word = FAST ? pack_bf16x2_cvt(lo, hi)
                                                       : f32_to_bf16_bits_rn(lo) | (f32_to_bf16_bits_rn(hi) << 16);
                            // streaming store: Y is not read again here, and
                            // evicting it first lets L2 write it back while
                            // the GEMM leaves HBM idle (1 % faster steps)
                            if (tk < ntok && fok) __stcs(reinterpret_cast<unsigned int *>(out + (size_t)tk * p.N), word);
                        }
                    }
                };
                if (fast_cvt) store_pairs(std::true_type{});
                else store_pairs(std::false_type{});
            }
        }
        __syncwarp();
    }
}

template <bool OUT_I32, bool GROUPED>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(THREADS, 1)
gemm_ts_kernel(const __grid_constant__ CUtensorMap tmX0, const __grid_constant__ CUtensorMap tmW0,
               const __grid_constant__ CUtensorMap tmX1, const __grid_constant__ CUtensorMap tmW1,
               const Params p) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t sb = (smem_addr(smem_raw) + 1023u) & ~1023u;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int pair = blockIdx.x >> 1;
    const int npairs = gridDim.x >> 1;

    if (threadIdx.x == 0) {
        for (int i = 0; i < S8; ++i) {
            mbar_init(sb + BAR_FULL8 + 8 * i, 1);
            mbar_init(sb + BAR_EMPTY8 + 8 * i, NUM_CONV_WARPS);
        }
        for (int i = 0; i < SA; ++i) {
            mbar_init(sb + BAR_SFULL + 8 * i, 2 * NUM_CONV_WARPS + 1);
            mbar_init(sb + BAR_SEMPTY + 8 * i, 1);
        }
        mbar_init(sb + BAR_ACCFULL, 1);
        mbar_init(sb + BAR_ACCEMPTY, 2 * NUM_EPI_WARPS);
        mbar_init(sb + BAR_DRAIN, 1);
        mbar_init(sb + BAR_TFLAG, 1);
        mbar_init(sb + BAR_TFLAG + 8, 1);
        st_shared_s32(sb + OFF_ABORT, 0);
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmX0);
        tma_prefetch_desc(&tmW0);
        tma_prefetch_desc(&tmX1);
        tma_prefetch_desc(&tmW1);
    }
    if (warp == 1) {
        tmem_alloc_pair(sb + OFF_TMEM, TMEM_COLS);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync();
    tc_fence_after();
    const uint32_t tmem = static_cast<uint32_t>(ld_shared_s32(sb + OFF_TMEM));
    const uint32_t peer_tmem = ld_shared_cluster_u32(mapa_shared(sb + OFF_TMEM, rank ^ 1u));
    const bool run_ok = (tmem == peer_tmem);
    if (!run_ok && threadIdx.x == 0) atomicOr(p.err, ERR_TMEM_PAIR);
    wait_prior_grid();
    const WaitCtx wc{sb + OFF_ABORT, p.err, p.wait_limit_ns};
    const int KB = p.k_blocks;                            // K=64 sub-blocks per tile
    const int NS = (KB + SUB - 1) / SUB;                  // stages per tile
    const int NC = (KB + KC_BLOCKS - 1) / KC_BLOCKS;      // chunks per tile

    if (warp >= 8) {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(REGS_HIGH));
        if (run_ok) epilogue_role<OUT_I32, GROUPED>(p, sb, tmem, wc, warp, lane, NC, rank, pair, npairs);
    } else {
        asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(REGS_LOW));
        if (!run_ok) {
        } else if (warp == 0) {
            // ------------------------------------------ TMA producer: weights
            if (lane == 0) {
                uint32_t j = 0;
                bool ok = true;
                for (int u = pair; ok && u < p.total_units; u += npairs) {
                    const Unit un = unit_coords(p, u, NC);
                    const Tile tl = tile_coords<GROUPED>(p, un.tile);
                    const CUtensorMap *mW = tl.branch ? &tmW1 : &tmW0;
                    const int frow = tl.f0 + static_cast<int>(rank) * CTA_F;
                    const int ks_end = min(NS, un.ci1 * KC_STAGES);
                    for (int ks = un.ci0 * KC_STAGES; ks < ks_end; ++ks, ++j) {
                        const uint32_t s = j % S8;
                        if (!mbar_wait(sb + BAR_EMPTY8 + 8 * s, ((j / S8) & 1) ^ 1, wc, ERR_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = sb + BAR_FULL8 + 8 * s;
                        const int nsub = min(SUB, KB - ks * SUB);     // the last stage may be half
                        mbar_arrive_expect_tx(fb, nsub * SUBW);
                        for (int u = 0; u < nsub; ++u)
                            tma_load_2d(sb + OFF_W + s * STAGE_W + u * SUBW, mW, (ks * SUB + u) * BK, frow, fb);
                    }
                }
                for (uint32_t i = (j > S8 ? j - S8 : 0); i < j; ++i)
                    mbar_wait(sb + BAR_FULL8 + 8 * (i % S8), (i / S8) & 1, wc, ERR_DRAIN, false);
            }
        } else if (warp == 2) {
            // -------------------------------------- TMA producer: activations
            // fp16 activation codes of this CTA's 128 tokens, straight into
            // the swizzled B operand; completion lands on the leader's
            // barrier, which the leader armed for both CTAs' bytes.  (Every
            // load has landed before the kernel ends: the MMA waits for each.)
            if (lane == 0) {
                uint32_t j = 0;
                bool ok = true;
                for (int u = pair; ok && u < p.total_units; u += npairs) {
                    const Unit un = unit_coords(p, u, NC);
                    const Tile tl = tile_coords<GROUPED>(p, un.tile);
                    const CUtensorMap *mX = tl.branch ? &tmX1 : &tmX0;
                    const int trow = tl.t0 + static_cast<int>(rank) * CTA_T;
                    const int ks_end = min(NS, un.ci1 * KC_STAGES);
                    for (int ks = un.ci0 * KC_STAGES; ks < ks_end; ++ks, ++j) {
                        const uint32_t s = j % SX;
                        if (!mbar_wait_cluster(sb + BAR_SEMPTY + 8 * s, ((j / SX) & 1) ^ 1, wc, ERR_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = mapa_shared(sb + BAR_SFULL + 8 * s, 0);
                        const int nsub = min(SUB, KB - ks * SUB);
                        if (leader) mbar_arrive_expect_tx(sb + BAR_SFULL + 8 * s, 2 * nsub * SUBX);
                        for (int u = 0; u < nsub; ++u)
                            tma_load_2d_pair(sb + OFF_X + s * STAGE_X + u * SUBX, mX, (ks * SUB + u) * BK, trow, fb);
                    }
                }
            }
        } else if (warp == 1) {
            // ------------------------------------------- MMA issue (leader)
            if (lane == 0 && leader) {
                constexpr uint32_t idesc = idesc_f16_f32(PAIR_F, PAIR_T);
                // the descriptor's start-address field is addr >> 4 in its
                // low 14 bits: offsets within the ring add without a carry
                const uint64_t b_desc0 = smem_desc_sw128(sb + OFF_X);
                static_assert(OFF_X + SX * STAGE_X <= (1u << 18), "descriptor start field");
                const uint32_t a_base = tmem + A_COL0;
                uint32_t j = 0, c = 0;         // stages, drains so far
                bool ok = true;
                const bool use_single = p.single_ok != 0;
                int n = 0;                     // units so far
                for (int u = pair; ok && u < p.total_units; u += npairs, ++n) {
                    const Unit un = unit_coords(p, u, NC);
                    const Tile tc = tile_coords<GROUPED>(p, un.tile);
                    const int fb = tc.f0 / PAIR_F;
                    const uint32_t *plan = p.br[tc.branch].plan;
                    bool single = false;       // the tile is one run (published by the epilogue)
                    bool fresh = true;         // the next MMA starts a new accumulation
                    for (int ci = un.ci0; ok && ci < un.ci1; ++ci) {
                        if (fresh) {
                            // the epilogue has drained the previous accumulation
                            if (!mbar_wait_cluster(sb + BAR_ACCEMPTY, (c & 1) ^ 1, wc, ERR_MMA)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                        }
                        const int ks0 = ci * KC_STAGES;
                        const int ks1 = min(NS, ks0 + KC_STAGES);
                        // one thread issues every MMA, at ~100 clk per
                        // instruction against 128 clk of tensor work each,
                        // so the per-stage bookkeeping is kept to a minimum:
                        // slot addresses and descriptors are offsets of
                        // values computed once, the accumulate flag is
                        // computed once per stage
                        static_assert(SA == 4 && SUB == 2, "slot arithmetic below");
                        for (int ks = ks0; ks < ks1; ++ks, ++j) {
                            const uint32_t sa = j & 3u;
                            if (!mbar_wait_cluster(sb + BAR_SFULL + 8 * sa, (j >> 2) & 1, wc, ERR_MMA)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            const uint32_t a = a_base + sa * A_SLOT_COLS;
                            const uint64_t bd = b_desc0 + sa * (STAGE_X >> 4);
                            const uint32_t acc = (!fresh || ks > ks0) ? 1u : 0u;
#pragma unroll
                            for (int kk = 0; kk < BK / 16; ++kk)
                                mma_f16_ts_pair(tmem, a + kk * 8, bd + kk * 2, idesc, kk > 0 ? 1u : acc);
                            if (ks * SUB + 1 < KB) {
#pragma unroll
                                for (int kk = 0; kk < BK / 16; ++kk)
                                    mma_f16_ts_pair(tmem, a + BK / 2 + kk * 8, bd + (SUBX >> 4) + kk * 2, idesc, 1u);
                            }
                            mma_commit_pair_multicast(sb + BAR_SEMPTY + 8 * sa, 0x3);
                        }
                        if (use_single && ci == un.ci0 && ok) {
                            if (!mbar_wait(sb + BAR_TFLAG + 8 * (n & 1), (n >> 1) & 1, wc, ERR_MMA)) {
                                ok = false;
                                break;
                            }
                            single = ld_shared_s32(sb + OFF_TFLAG + 4 * (n & 1)) != 0;
                        }
                        fresh = ci == un.ci1 - 1 || (!single && plan_drains(p, plan, fb, ci, NC));
                        if (ok && fresh) {
                            mma_commit_pair_multicast(sb + BAR_ACCFULL, 0x3);
                            ++c;
                        }
                    }
                }
                mma_commit_pair(sb + BAR_DRAIN);
                mbar_wait_cluster(sb + BAR_DRAIN, 0, wc, ERR_DRAIN, false);
            }
        } else if (warp >= 4) {
            // ---------------------------------------------------- converters
            // thread = weight row r of this CTA = TMEM lane r; each K=64
            // sub-block of the row is 64 bytes in four 16-byte chunks, chunk
            // c at c ^ ((r >> 1) & 3) (the 64-byte swizzle, which spreads 8
            // consecutive rows over all banks)
            const uint32_t r = static_cast<uint32_t>((warp & 3) * 32 + lane);
            const uint32_t src_row = r * BK;
            const uint32_t sw = (r >> 1) & 3;
            const uint32_t a_lane = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16) + A_COL0;
            uint32_t j = 0;
            bool ok = true;
            for (int u = pair; ok && u < p.total_units; u += npairs) {
                const Unit un = unit_coords(p, u, NC);
                const int ks_end = min(NS, un.ci1 * KC_STAGES);
                for (int ks = un.ci0 * KC_STAGES; ks < ks_end; ++ks, ++j) {
                    const uint32_t s8 = j % S8, sa = j % SA;
                    // every lane waits; __all_sync keeps the warp's control flow
                    // uniform if a wait gives up
                    if (!__all_sync(0xffffffffu, mbar_wait(sb + BAR_FULL8 + 8 * s8, (j / S8) & 1, wc,
                                                            ERR_CONVERTER))) {
                        ok = false;
                        break;
                    }
                    const uint32_t src = sb + OFF_W + s8 * STAGE_W + src_row;
                    uint4 v[4];
#pragma unroll
                    for (int cc = 0; cc < 4; ++cc) v[cc] = ld_shared_v4(src + ((cc ^ sw) << 4));
                    if (!__all_sync(0xffffffffu, mbar_wait_cluster(sb + BAR_SEMPTY + 8 * sa, ((j / SA) & 1) ^ 1,
                                                                    wc, ERR_CONVERTER))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    // convert sub-block u (its codes in v) and write it into
                    // the slot's columns 32u .. 32u + 31
                    auto convert_store = [&](int u) {
                        uint32_t w[32];
#pragma unroll
                        for (int cc = 0; cc < 4; ++cc) {
                            i8x4_to_f16x4(v[cc].x, w[8 * cc + 0], w[8 * cc + 1]);
                            i8x4_to_f16x4(v[cc].y, w[8 * cc + 2], w[8 * cc + 3]);
                            i8x4_to_f16x4(v[cc].z, w[8 * cc + 4], w[8 * cc + 5]);
                            i8x4_to_f16x4(v[cc].w, w[8 * cc + 6], w[8 * cc + 7]);
                        }
                        tmem_st_32x32b_x32(a_lane + sa * A_SLOT_COLS + u * (BK / 2), w);
                    };
                    static_assert(SUB == 2, "two sub-blocks per stage");
                    convert_store(0);
                    if (ks * SUB + 1 < KB) {            // the last stage may be half
                        // loaded once sub-block 0's codes are out of the way
#pragma unroll
                        for (int cc = 0; cc < 4; ++cc) v[cc] = ld_shared_v4(src + SUBW + ((cc ^ sw) << 4));
                        convert_store(1);
                    }
                    // the stage's bytes are all in registers (and in TMEM) now
                    __syncwarp();
                    if (lane == 0) mbar_arrive(sb + BAR_EMPTY8 + 8 * s8);
                    tmem_st_wait();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) arrive_leader(sb + BAR_SFULL + 8 * sa, rank);
                }
            }
        }
    }
    tc_fence_before();
    __syncwarp();
    asm volatile("bar.sync 1, %0;" ::"n"(THREADS) : "memory");
    cluster_sync();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, TMEM_COLS);
    }
}

// ------------------------------------------------------------ drain plan
//
// The fixed chunk of 1024 products is the worst case (every |a|, |w| at its
// maximum).  A tighter bound holds per weight row: every partial sum that
// the tensor core forms over a K range is at most sum |a_k| |w_k| <=
// 128 * sum |w_k| over that range (|a| <= 128 for an int8 code), so runs of
// chunks whose weight rows all have sum |w_k| <= 2^17 keep every partial sum
// within 2^24, exact in fp32, and need no drain in between.  The plan is
// built once per weight matrix: per block of 256 rows (one tile of the GEMM),
// chunks are merged greedily while the largest row's sum over the merged run
// stays within the bound.  A block's last word holds the largest sum of
// squares of its rows, for the bound that uses the activations too (see
// tile_single_run).
constexpr uint32_t kPlanL1Limit = 1u << 17;
constexpr int KC = KC_BLOCKS * BK;                   // K per chunk

__global__ void __launch_bounds__(PAIR_F)
chunk_plan_kernel(const int8_t *__restrict__ Wq, int N, int K, int NC, int words, uint32_t *__restrict__ plan) {
    __shared__ uint32_t red[PAIR_F / 32];
    const int fb = blockIdx.x;
    const int r = fb * PAIR_F + threadIdx.x;
    uint32_t *row_plan = plan + (size_t)fb * (words + 1);
    if (threadIdx.x == 0)
        for (int w = 0; w < words; ++w) row_plan[w] = 0u;
    uint32_t cur = 0;                                 // this row's sum |w| since the last drain
    uint32_t sq = 0;                                  // this row's sum of squares (< 2^32: K * 127^2)
    for (int c = 0; c < NC; ++c) {
        uint32_t l1 = 0;
        if (r < N) {
            const int k1 = min(K, (c + 1) * KC);
            const uint4 *src = reinterpret_cast<const uint4 *>(Wq + (size_t)r * K);
            for (int k = c * KC; k < k1; k += 16) {
                const uint4 v = __ldg(src + k / 16);
                const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const uint32_t a4 = __vabsdiffs4(w4[e], 0u);
                    l1 = __dp4a(a4, 0x01010101u, l1);
                    sq = __dp4a(a4, a4, sq);
                }
            }
        }
        const uint32_t cand = cur + l1;
        const uint32_t wm = __reduce_max_sync(0xffffffffu, cand);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = wm;
        __syncthreads();
        uint32_t m = 0;
#pragma unroll
        for (int w = 0; w < PAIR_F / 32; ++w) m = max(m, red[w]);
        __syncthreads();
        if (m > kPlanL1Limit) {                       // chunk c starts a new run
            if (threadIdx.x == 0) row_plan[(c - 1) >> 5] |= 1u << ((c - 1) & 31);
            cur = l1;
        } else {
            cur = cand;
        }
    }
    const uint32_t wm = __reduce_max_sync(0xffffffffu, sq);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = wm;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t m = 0;
#pragma unroll
        for (int w = 0; w < PAIR_F / 32; ++w) m = max(m, red[w]);
        row_plan[words] = m;
        row_plan[(NC - 1) >> 5] |= 1u << ((NC - 1) & 31);
    }
}

// ------------------------------------------ int8 codes into this engine
//
// The int8 codes that a3 writes (w8a8_quant_act) reach this engine through
// one streaming pass: each warp takes one token row, reads its codes 8 per
// lane (256 bytes per warp instruction), writes them as fp16 values (the
// weights' conversion; 512 bytes per store instruction) and sums their
// squares exactly with dp4a: |code| <= 128 and K < 2^18 keep every sum
// below 2^32, and the int32 adds wrap like the uint32 ones.  The fp16 codes
// (2MK bytes) are written back into L2, where the GEMM that follows finds
// them.  One launch covers both branches of a dual call: rows [0, M0) are
// branch 0's, the rest branch 1's.
struct ExpandBranch {
    const int8_t *Xq;
    uint16_t *Xq16;
    uint32_t *sumsq;
    int M;
};

constexpr int kExpandThreads = 256;
constexpr int kExpandBatch = 16;                      // 8-code loads in flight per lane

__global__ void __launch_bounds__(kExpandThreads)
expand_codes_kernel(const __grid_constant__ ExpandBranch b0, const __grid_constant__ ExpandBranch b1, int K) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int lane = threadIdx.x & 31;
    // one warp per row, the row index in 64 bits (the grid grows with M0 + M1)
    long long r = (static_cast<long long>(blockIdx.x) * kExpandThreads + threadIdx.x) >> 5;
    const bool second = r >= b0.M;
    const ExpandBranch &b = second ? b1 : b0;
    if (second) r -= b0.M;
    if (r >= b.M) return;                             // whole warps leave together
    const int row = static_cast<int>(r);
    const int n8 = K / 8;                             // 8-code groups per row
    const uint2 *src = reinterpret_cast<const uint2 *>(b.Xq + (size_t)row * K);
    uint4 *dst = reinterpret_cast<uint4 *>(b.Xq16 + (size_t)row * K);
    int ss = 0;
    for (int g0 = 0; g0 < n8; g0 += 32 * kExpandBatch) {
        uint2 v[kExpandBatch];
#pragma unroll
        for (int i = 0; i < kExpandBatch; ++i) {
            const int g = g0 + i * 32 + lane;
            v[i] = g < n8 ? __ldcs(src + g) : make_uint2(0u, 0u);
        }
#pragma unroll
        for (int i = 0; i < kExpandBatch; ++i) {
            const int g = g0 + i * 32 + lane;
            if (g < n8) {
                uint4 o;
                i8x4_to_f16x4(v[i].x, o.x, o.y);
                i8x4_to_f16x4(v[i].y, o.z, o.w);
                dst[g] = o;
                ss = __dp4a(static_cast<int>(v[i].x), static_cast<int>(v[i].x), ss);
                ss = __dp4a(static_cast<int>(v[i].y), static_cast<int>(v[i].y), ss);
            }
        }
    }
    const uint32_t t = __reduce_add_sync(0xffffffffu, static_cast<uint32_t>(ss));
    if (lane == 0) b.sumsq[row] = t;
}

// ------------------------------------------------------------------ host

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode() {
    // a function-local static: initialised once, thread-safe
    static const EncodeTiledFn fn = [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<EncodeTiledFn>(ptr);
        return static_cast<EncodeTiledFn>(nullptr);
    }();
    return fn;
}

// row-major [rows, inner] -> 2-D map with box [box_rows, box_inner], zero fill
bool make_map(CUtensorMap *m, CUtensorMapDataType dt, const void *base, uint64_t inner, uint64_t rows,
              uint64_t row_bytes, uint32_t box_inner, uint32_t box_rows, CUtensorMapSwizzle sw) {
    EncodeTiledFn enc = get_encode();
    if (!enc) return false;
    cuuint64_t dims[2] = {inner, rows};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_rows};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, dt, 2, const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Per variant and device: the dynamic shared memory limit set and the
// registers ptxas gave the kernel (the register split assumes exactly
// LAUNCH_REGS at launch).
template <bool OUT_I32, bool GROUPED>
cudaError_t prepare_ts_kernel() {
    static PerDevice<int> regs;
    int n = 0;
    cudaError_t e = regs.get([](int &v) {
        cudaFuncAttributes fa;
        cudaError_t r = cudaFuncGetAttributes(&fa, gemm_ts_kernel<OUT_I32, GROUPED>);
        if (r != cudaSuccess) return r;
        v = fa.numRegs;
        return cudaFuncSetAttribute(gemm_ts_kernel<OUT_I32, GROUPED>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_TOTAL);
    }, &n);
    if (e != cudaSuccess) return e;
    return n == LAUNCH_REGS ? cudaSuccess : cudaErrorInvalidConfiguration;
}

}  // namespace

int chunk_plan_bits_words(int K) {
    const int NC = (K + KC - 1) / KC;
    return (NC + 31) / 32;
}

int chunk_plan_words(int K) { return chunk_plan_bits_words(K) + 1; }

cudaError_t launch_chunk_plan(const int8_t *Wq, int N, int K, uint32_t *plan, cudaStream_t st) {
    const int NC = (K + KC - 1) / KC;
    chunk_plan_kernel<<<(N + PAIR_F - 1) / PAIR_F, PAIR_F, 0, st>>>(Wq, N, K, NC, chunk_plan_bits_words(K), plan);
    return cudaGetLastError();
}

// Split-K workspace: the arrival counters (16 per split tile: one per
// epilogue warp of each CTA), then one int32 partial tile per split part.  A
// launch splits at most as many parts as there are CTA pairs.
namespace {
constexpr size_t kWsCounterBytes(int pairs) { return ((size_t)pairs * 16 * 4 + 255) / 256 * 256; }
constexpr int kSplitMaxRounds = 12;
}  // namespace

long long gemm_ts_workspace_bytes() {
    const int P = device_sms() / 2;
    return static_cast<long long>(kWsCounterBytes(P) + (size_t)P * PAIR_T * PAIR_F * 4);
}

cudaError_t launch_gemm_ts(const GemmBranch *br, int nb, int N, int K, bool out_i32, void *workspace,
                           unsigned int *err, cudaStream_t st) {
    const int sms = device_sms();
    Params p{};
    CUtensorMap maps[4];
    int first = -1;
    const int f_tiles = (N + PAIR_F - 1) / PAIR_F;
    for (int i = 0; i < 2; ++i) {
        const GemmBranch *b = (i < nb) ? &br[i] : nullptr;
        BranchArgs &a = p.br[i];
        a = BranchArgs{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, 0, 0, 0};
        if (b && b->M > 0) {
            a.x_scale = b->x_scale;
            a.w_scale = b->w_scale;
            a.bias = b->bias;
            a.out = b->out;
            a.x_sumsq = b->x_sumsq;
            a.plan = b->plan;
            a.M = b->M;
            a.t_tiles = (b->M + PAIR_T - 1) / PAIR_T;
            a.tiles = a.t_tiles * f_tiles;
            if (!make_map(&maps[2 * i], CU_TENSOR_MAP_DATA_TYPE_FLOAT16, b->Xq, K, b->M, 2ull * K, BK, CTA_T,
                          CU_TENSOR_MAP_SWIZZLE_128B) ||
                !make_map(&maps[2 * i + 1], CU_TENSOR_MAP_DATA_TYPE_UINT8, b->Wq, K, N, K, BK, CTA_F,
                          CU_TENSOR_MAP_SWIZZLE_64B))
                return cudaErrorInvalidValue;
            if (first < 0) first = i;
        }
    }
    if (first < 0) return cudaSuccess;
    for (int i = 0; i < 2; ++i)
        if (p.br[i].M == 0) {
            maps[2 * i] = maps[2 * first];
            maps[2 * i + 1] = maps[2 * first + 1];
        }
    p.N = N;
    p.K = K;
    p.total_tiles = p.br[0].tiles + p.br[1].tiles;
    // tile order (tile_order.cuh): the codes are 2 bytes, the weights 1
    p.f_tiles = f_tiles;
    p.group_f = tile_group(2LL * K * (p.br[0].M > p.br[1].M ? p.br[0].M : p.br[1].M),
                           static_cast<long long>(PAIR_F) * K, f_tiles);
    p.k_blocks = (K + BK - 1) / BK;
    p.plan_words = chunk_plan_words(K);
    p.single_ok = 1;
    for (int i = 0; i < 2; ++i)
        if (p.br[i].M > 0 && (p.br[i].x_sumsq == nullptr || p.br[i].plan == nullptr)) p.single_ok = 0;
    p.err = err;
    p.wait_limit_ns = 2000000000ull;
    // The tiles fill the CTA pairs in rounds; a last, partial round would
    // leave pairs idle, so with a workspace R = T mod pairs tiles are split
    // into s parts of consecutive K chunks (s R <= pairs, s <= chunks), one
    // part per pair, run in the first round.  With fewer tiles than pairs,
    // every tile is split.  It saves at most one round of T / pairs + 1, so
    // it is used only up to kSplitMaxRounds full rounds: beyond that the
    // exchange of partial sums costs more than the round it saves (measured:
    // 1280 tokens +10 %, 4608 +3 %, 16896 -2.5 % on the DiT block's GEMMs).
    const int P = sms / 2;
    const int T = p.total_tiles;
    const int NC = (K + KC - 1) / KC;
    p.full_tiles = T;
    p.split = 1;
    p.split_tiles = 0;
    if (workspace != nullptr && NC >= 2 && T / P <= kSplitMaxRounds) {
        const int rem = T % P;
        const int s = rem > 0 ? min(P / rem, NC) : 1;
        if (s >= 2) {
            p.full_tiles = T - rem;
            p.split = s;
            p.split_tiles = rem;
            p.ws_cnt = static_cast<unsigned int *>(workspace);
            p.ws = reinterpret_cast<int32_t *>(static_cast<char *>(workspace) + kWsCounterBytes(P));
        }
    }
    p.total_units = p.full_tiles + p.split_tiles * p.split;
    const int pairs = p.total_units < P ? p.total_units : P;
    const bool grouped = p.group_f > 1;
    auto kern = out_i32 ? (grouped ? gemm_ts_kernel<true, true> : gemm_ts_kernel<true, false>)
                        : (grouped ? gemm_ts_kernel<false, true> : gemm_ts_kernel<false, false>);
    cudaError_t e = out_i32 ? (grouped ? prepare_ts_kernel<true, true>() : prepare_ts_kernel<true, false>())
                            : (grouped ? prepare_ts_kernel<false, true>() : prepare_ts_kernel<false, false>());
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(2 * pairs), THREADS, SMEM_TOTAL, st, maps[0], maps[1], maps[2], maps[3], p);
}

// The int8-code linear on this engine.  Workspace layout: the split-K area
// (gemm_ts_workspace_bytes(), first, so that its counters stay where the
// caller zeroed them), then each branch's fp16 codes and each branch's
// token sums, every piece starting on a 256-byte boundary.
namespace {
constexpr size_t round256(size_t n) { return (n + 255) / 256 * 256; }
}  // namespace

long long linear_codes8_workspace_bytes(long long tokens, int K) {
    if (tokens < 0 || K <= 0) return 0;
    return gemm_ts_workspace_bytes() + 2 * tokens * K + 4 * tokens + 4 * 256;
}

void linear_workspace_views(void *workspace, int M, int K, uint16_t **codes16, uint32_t **sumsq) {
    char *w = static_cast<char *>(workspace);
    const size_t off = static_cast<size_t>(gemm_ts_workspace_bytes());
    *codes16 = reinterpret_cast<uint16_t *>(w + off);
    *sumsq = reinterpret_cast<uint32_t *>(w + off + round256(2 * static_cast<size_t>(M) * K));
}

cudaError_t launch_linear_codes8(const GemmBranch *br, int nb, int N, int K, bool out_i32, void *workspace,
                                 unsigned int *err, cudaStream_t st) {
    char *w = static_cast<char *>(workspace);
    size_t off = static_cast<size_t>(gemm_ts_workspace_bytes());
    ExpandBranch eb[2] = {{nullptr, nullptr, nullptr, 0}, {nullptr, nullptr, nullptr, 0}};
    GemmBranch gb[2];
    for (int i = 0; i < nb; ++i) {
        gb[i] = br[i];
        if (br[i].M <= 0) continue;
        eb[i].Xq = br[i].Xq;
        eb[i].M = br[i].M;
        eb[i].Xq16 = reinterpret_cast<uint16_t *>(w + off);
        off += round256(2 * static_cast<size_t>(br[i].M) * K);
    }
    for (int i = 0; i < nb; ++i) {
        if (br[i].M <= 0) continue;
        eb[i].sumsq = reinterpret_cast<uint32_t *>(w + off);
        off += round256(4 * static_cast<size_t>(br[i].M));
        gb[i].Xq = reinterpret_cast<const int8_t *>(eb[i].Xq16);
        gb[i].x_sumsq = eb[i].sumsq;
    }
    const long long rows = static_cast<long long>(eb[0].M) + eb[1].M;
    if (rows == 0) return cudaSuccess;
    const int rows_per_block = kExpandThreads / 32;
    const long long blocks = (rows + rows_per_block - 1) / rows_per_block;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
    expand_codes_kernel<<<static_cast<unsigned int>(blocks), kExpandThreads, 0, st>>>(eb[0], eb[1], K);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return launch_gemm_ts(gb, nb, N, K, out_i32, workspace, err, st);
}

}  // namespace w8a8
