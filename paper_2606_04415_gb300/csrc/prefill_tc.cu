// Prefill attention on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// Prefill is the compute-bound phase (Sec. 1, Sec. 3.3, Fig. 1): QK^T and PV
// are dense bf16 contractions, so they run as tcgen05.mma with fp32
// accumulators in tensor memory.
//
// GQA packing: a Q tile is 128 MMA rows = (position, query head) pairs of one
// kv head (row = p * G + h, P = floor(128 / G) positions), so each K/V byte
// staged in shared memory serves all G heads of the group (126 of 128 rows
// busy for G = 7). A 3-D TMA box (64 columns x G heads x P positions) writes
// exactly this row order. A work item is two consecutive Q tiles of one kv
// head (2P positions) that consume the same K/V tiles, which halves the
// L2-to-SM traffic per FLOP.
//
// Key tiles are 128 keys wide: an S = Q K^T product is then M = N = 128 and
// runs at the full tensor rate (a 64-wide one, with both operands in shared
// memory, is bound by shared-memory bandwidth: 48 instead of 32 cycles).
//
// One persistent CTA per SM (384 threads) takes items, longest first, from an
// atomic queue (the last CTA to finish resets it for the next run):
//   warps 0-3, 4-7  softmax warpgroups for Q tile 0 and tile 1, one MMA row
//                   per thread: the 128 scores of the row from TMEM into
//                   registers, online softmax, P (bf16) written back over the
//                   first 64 columns of S, lazy rescale of the O row,
//                   epilogue;
//   warp 8          scheduler and K producer: the item's two Q tiles, then the
//                   128-key K tiles gathered block by block through the block
//                   table (one 4-D box per block and 64-column half) into a
//                   3-stage ring;
//   warp 9          V producer (2-stage ring); zeroes V rows past the context
//                   before the last PV of an item;
//   warp 10         issues every MMA, in the order PV_0(j), S_0(j+1), PV_1(j),
//                   S_1(j+1): the tensor pipe completes a thread's MMAs in
//                   issue order, so S_w(j+1) overwrites P_w(j) only after
//                   PV_w(j) has read it, and when S_w(j) is complete so is
//                   PV_w(j-1) -- the softmax may rescale O_w at that point
//                   without a further wait. With a single V stage (192-wide
//                   keys) the order is PV_0(j), PV_1(j), S_0(j+1), S_1(j+1),
//                   so that V(j+1) loads while both S of the next tile run.
// TMEM (512 columns): S0 at 0, S1 at 128 (fp32, P over their first 64
// columns); O0 at 256, O1 at 384.
// Every mbarrier wait is bounded; a timeout raises the plan's error flag and
// the CTA drains its tensor-core work, frees its tensor memory and exits.
// Launched as a programmatic dependent of the kernel before it (the step's
// KV append), the grid sets up while that kernel drains; the two loader
// warps wait for it (griddepcontrol.wait) before their first read, and every
// other warp reads global memory only after them. Optionally (a cooperative
// launch, fused_append) the CTAs write the step's prefill rows into the cache
// themselves first and wait for one another before any warp takes its role.
#include <math.h>

#include "common.cuh"
#include "fp8.cuh"
#include "tc.cuh"

namespace fnpu {
namespace {

constexpr int kThreads = 384;
constexpr int kRows = 128;
constexpr int kKeys = 128;   // keys per tile
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: p <= 2^8 before a rescale
// Register split (setmaxnreg): the softmax warpgroups hold a 128-score row
// each; the producer and MMA warpgroup needs few.
constexpr uint32_t kRegsSoftmax = 208;
constexpr uint32_t kRegsHelper = 88;
static_assert(2 * 128 * kRegsSoftmax + 128 * kRegsHelper <= 65536 / kThreads / 8 * 8 * kThreads, "register split");

__host__ __device__ constexpr uint32_t col_s(int w) { return 128u * w; }
__host__ __device__ constexpr uint32_t col_o(int w) { return 256u + 128u * w; }

// DQ: key (and query) width, DV: value width. 128-wide keys take a 3-stage K
// ring and a 2-stage V ring; 192-wide keys (MLA rows expanded per head) leave
// shared memory for 2 K stages and 1 V stage beside the two Q tiles.
template <int DQ, int DV>
struct TcCfg {
    static_assert(DQ % 64 == 0 && DV % 64 == 0 && DV <= 128, "tile widths");
    static constexpr int kKStages = DQ > 128 ? 2 : 3;  // K ring
    static constexpr int kVStages = DQ > 128 ? 1 : 2;  // V ring
    static constexpr int kKTileBytes = kKeys * DQ * 2;  // one K tile
    static constexpr int kVTileBytes = kKeys * DV * 2;  // one V tile
    static constexpr int kHalf = kKeys * 128;           // one 64-column chunk of a K/V tile
    static constexpr int kQHalf = kRows * 128;          // one 64-column chunk of a Q tile
    static constexpr int kQBytes = kRows * DQ * 2;      // one Q tile
    static constexpr int kVOff = kKStages * kKTileBytes;
    static constexpr int kQOff = kVOff + kVStages * kVTileBytes;
    static constexpr int kBarOff = kQOff + 2 * kQBytes;
    // kfull[3] kempty[3] vfull[2] vempty[2] sfull[2] pfull[2] odone[2] ofree[2]
    // qfull qempty vzero itemfull[2] itemempty[2] drain
    static constexpr int kNumBars = 2 * kKStages + 2 * kVStages + 8 + 3 + 4 + 1;
    static constexpr int kSmemUsed = kBarOff + 8 * kNumBars + 32;
    // at least 116 KB so that no two CTAs share an SM (each holds all 512 TMEM columns)
    static constexpr int kSmemBytes = kSmemUsed > 116 * 1024 ? kSmemUsed : 116 * 1024;
    static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
};

struct TcMaps {
    CUtensorMap k, v, q;
};

struct ItemGeom {
    int kvh, p0, rows, prefix, ctx, kt0, ntiles, q_start, bt_row;
    int ns, split, pbase, cnt;  // key splits of the tile pair, this split, first partial, merge counter
    bool tail_fix;
};

__device__ __forceinline__ ItemGeom item_geom(const AttnParams &p, int idx) {
    const PrefillItem it = p.pitems[idx];  // carries its sequence's fields: one load
    ItemGeom g;
    g.kvh = it.head;
    g.p0 = it.row_begin;
    g.rows = it.rows;
    g.prefix = it.prefix;
    g.ctx = it.ctx_len;
    g.kt0 = it.kt_begin;              // 128-key tiles [kt_begin, kt_end) of keys 0 .. last position
    g.ntiles = it.kt_end - it.kt_begin;
    g.q_start = it.q_start;
    g.bt_row = it.bt_row;
    g.ns = it.num_splits;
    g.split = it.split;
    g.pbase = it.part_base;
    g.cnt = it.group;
    g.tail_fix = it.kt_end * kKeys > g.ctx;
    return g;
}

// The step's append of the prefill-path rows inside the prefill grid
// (fnpu_mixed_step; both phases share the KV pool, Sec. 3.4), shared by the
// CTAs: 16-byte chunks, consecutive threads on consecutive chunks of a row,
// the row and its slot loaded together. Then every CTA waits (bounded) until
// all have written theirs, before any warp reads the cache; the launch is
// cooperative, so all are resident. False if the wait ran out (the plan's
// error flag is raised). A call of its own, so that the kernel's warps keep
// their register allocation.
__device__ __noinline__ bool fused_append(const AttnParams &p, int tid) {
    const int32_t kc = p.fa_k_chunks, per_tok = kc + p.fa_v_chunks;
    const int64_t total = static_cast<int64_t>(p.fa_num_tokens) * per_tok;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + tid; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int32_t ti = static_cast<int32_t>(i / per_tok);
        const int32_t c = static_cast<int32_t>(i - static_cast<int64_t>(ti) * per_tok);
        const int64_t t = __ldg(p.fa_tokens + ti);
        const uint4 v = c < kc ? __ldg(p.fa_k_new + t * kc + c) : __ldg(p.fa_v_new + t * p.fa_v_chunks + (c - kc));
        const int64_t s = __ldg(p.fa_slots + t);
        if (s < 0) continue;  // padding
        if (s >= p.fa_num_slots) {
            if (c == 0) atomicOr(p.fa_range_err, 1);
            continue;
        }
        if (c < kc) p.fa_k_cache[s * kc + c] = v;
        else p.fa_v_cache[s * p.fa_v_chunks + (c - kc)] = v;
    }
    tc::fence_proxy_async_global();  // before the TMA reads of the rows, here and in other CTAs
    __syncthreads();
    __shared__ int ok_all;
    if (tid == 0) {
        __threadfence();
        atomicAdd(p.fa_count, 1);
        int spins = 0, ok = 1;
        while (tc::ld_acquire_gpu(p.fa_count) < static_cast<int>(gridDim.x)) {
            if (++spins > (1 << 22)) {  // a CTA that never came: flag it, and leave the work undone
                atomicOr(p.err, 1);
                ok = 0;
                break;
            }
            __nanosleep(32);
        }
        tc::fence_proxy_async_global();
        ok_all = ok;
    }
    __syncthreads();
    return ok_all != 0;
}

// F16: the operands (Q, K, V and P) are f16 instead of bf16 (the FP8 cache's
// prefill: its codes are dequantised to f16 first)
template <int DQ, int DV, bool F16>
__global__ void __launch_bounds__(kThreads, 1)
    prefill_tc_kernel(const AttnParams p, const __grid_constant__ TcMaps maps) {
    using Cfg = TcCfg<DQ, DV>;
    constexpr int kKStages = Cfg::kKStages, kVStages = Cfg::kVStages;
    extern __shared__ __align__(1024) uint8_t smem[];
    const uint32_t s_base = smem_u32(smem);
    const uint32_t s_bars = s_base + Cfg::kBarOff;
    auto KFULL = [&](int s) { return s_bars + 8 * s; };
    auto KEMPTY = [&](int s) { return s_bars + 8 * (kKStages + s); };
    auto VFULL = [&](int s) { return s_bars + 8 * (2 * kKStages + s); };
    auto VEMPTY = [&](int s) { return s_bars + 8 * (2 * kKStages + kVStages + s); };
    const uint32_t b0 = s_bars + 8 * (2 * kKStages + 2 * kVStages);
    auto SFULL = [&](int w) { return b0 + 8 * w; };
    auto PFULL = [&](int w) { return b0 + 16 + 8 * w; };
    auto ODONE = [&](int w) { return b0 + 32 + 8 * w; };
    auto OFREE = [&](int w) { return b0 + 48 + 8 * w; };
    const uint32_t QFULL = b0 + 64, QEMPTY = b0 + 72, VZERO = b0 + 80;
    auto ITEMFULL = [&](int k) { return b0 + 88 + 8 * k; };
    auto ITEMEMPTY = [&](int k) { return b0 + 104 + 8 * k; };
    const uint32_t DRAIN = b0 + 120;
    uint8_t *misc = smem + Cfg::kBarOff + 8 * Cfg::kNumBars;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(misc);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc + 4);
    volatile int *item_slot = reinterpret_cast<volatile int *>(misc + 8);  // [2]

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = p.group;
    const int P = kRows / G;
    if ((s_base & 1023u) != 0) {  // the swizzled tiles need 1024-byte alignment
        if (tid == 0) atomicOr(p.err, 2);
        return;
    }

    if (tid == 0) {
        for (int s = 0; s < kKStages; ++s) {
            tc::mbar_init(KFULL(s), 1);
            tc::mbar_init(KEMPTY(s), 1);
        }
        for (int s = 0; s < kVStages; ++s) {
            tc::mbar_init(VFULL(s), 1);
            tc::mbar_init(VEMPTY(s), 1);
        }
        for (int w = 0; w < 2; ++w) {
            tc::mbar_init(SFULL(w), 1);
            tc::mbar_init(PFULL(w), kRows);
            tc::mbar_init(ODONE(w), 1);
            tc::mbar_init(OFREE(w), kRows);
            tc::mbar_init(ITEMFULL(w), 1);
            tc::mbar_init(ITEMEMPTY(w), 2 + 2 * kRows);  // MMA issuer, V producer, 256 softmax rows
        }
        tc::mbar_init(QFULL, 1);
        tc::mbar_init(QEMPTY, 1);
        tc::mbar_init(VZERO, 1);
        tc::mbar_init(DRAIN, 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
    }
    if (warp == 0) {
        tc::tmem_alloc(smem_u32(const_cast<uint32_t *>(tmem_slot)), kTmemCols);
        tc::tmem_relinquish();
    }
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *tmem_slot;

    if (p.fa_count != nullptr && !fused_append(p, tid)) *abort_flag = 1;

    auto wait = [&](uint32_t bar, uint32_t parity) -> bool {
        if (tc::mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (tc::mbar_wait(bar, parity)) return true;
        *abort_flag = 1;
        atomicOr(p.err, 1);
        return false;
    };

    if (warp >= 8) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(kRegsHelper));
    if (warp == 8 || warp == 9) {
        pdl_wait();  // the cache writes of the kernel before (the step's append)
        // ---------------------------------- producers (8: scheduler, Q, K; 9: V)
        const bool is_k = warp == 8;
        if (lane == 0) {
            tc::prefetch_tmap(is_k ? &maps.k : &maps.v);
            if (is_k) tc::prefetch_tmap(&maps.q);
        }
        const int bs = p.block_size;
        const int per_tile = kKeys / bs;  // blocks per tile (<= 8)
        const int nst = is_k ? kKStages : kVStages;
        const CUtensorMap *map = is_k ? &maps.k : &maps.v;
        int g = 0;  // tiles issued so far (ring position)
        int nfix = 0;
        for (int k = 0;; ++k) {
            const int slot = k & 1;
            int idx = 0;
            if (is_k) {
                // the first item of CTA b is item b (the queue hands the first
                // gridDim.x items out in that order anyway); later ones come
                // from the queue
                if (lane == 0) idx = k == 0 ? static_cast<int>(blockIdx.x) : static_cast<int>(gridDim.x) + atomicAdd(p.sched, 1);
                idx = __shfl_sync(0xffffffffu, idx, 0);
                if (k >= 2 && !wait(ITEMEMPTY(slot), ((k >> 1) - 1) & 1)) break;
                if (lane == 0) {
                    item_slot[slot] = idx < p.num_pitems ? idx : -1;
                    tc::mbar_arrive(ITEMFULL(slot));
                }
                if (idx >= p.num_pitems) break;
            } else {
                if (!wait(ITEMFULL(slot), (k >> 1) & 1)) break;
                idx = __shfl_sync(0xffffffffu, item_slot[slot], 0);
                if (idx < 0) break;
            }
            const ItemGeom it = item_geom(p, idx);
            const int ukvh = __shfl_sync(0xffffffffu, it.kvh, 0);
            // both Q tiles, once the previous item's last S is done (loading them
            // after the item's first K tiles, with an L2 prefetch ahead, was
            // measured slower)
            const int q0 = __shfl_sync(0xffffffffu, it.q_start + it.p0, 0);
            auto load_q = [&]() -> bool {
                if (k >= 1 && !wait(QEMPTY, (k - 1) & 1)) return false;
                tc::mbar_arrive_expect_tx_warp(QFULL, static_cast<uint32_t>(2 * (DQ / 64) * 64 * G * P * 2));
#pragma unroll
                for (int w = 0; w < 2; ++w)
#pragma unroll
                    for (int h = 0; h < DQ / 64; ++h)
                        tc::tma_load_3d_warp(s_base + Cfg::kQOff + w * Cfg::kQBytes + h * Cfg::kQHalf, &maps.q,
                                             QFULL, h * 64, ukvh * G, q0 + w * P);
                return true;
            };
            const int32_t *bt = p.block_table + static_cast<int64_t>(it.bt_row) * p.bt_stride;
            const int nblk_seq = (it.ctx + bs - 1) / bs;
            // block ids of the next tile, one per lane, loaded a tile ahead so
            // that the TMA issue never waits on a block-table read
            const int b00 = it.kt0 * per_tile;
            int blk_next = (lane < per_tile && b00 + lane < nblk_seq) ? __ldg(bt + b00 + lane) : 0;
            bool ok = true;
            for (int i = 0; i < it.ntiles; ++i, ++g) {
                if (is_k && i == 0 && !load_q()) { ok = false; break; }
                const int st = g % nst;
                const int blk_cur = blk_next;
                const int jn = b00 + (i + 1) * per_tile + lane;
                blk_next = (i + 1 < it.ntiles && lane < per_tile && jn < nblk_seq) ? __ldg(bt + jn) : 0;
                if (g >= nst && !wait(is_k ? KEMPTY(st) : VEMPTY(st), ((g / nst) - 1) & 1)) { ok = false; break; }
                int nvalid = nblk_seq - b00 - i * per_tile;
                nvalid = nvalid < 0 ? 0 : (nvalid > per_tile ? per_tile : nvalid);
                nvalid = __shfl_sync(0xffffffffu, nvalid, 0);
                const uint32_t bar = is_k ? KFULL(st) : VFULL(st);
                if constexpr (DQ == DV) {
                    const uint32_t dst = s_base + (is_k ? 0 : Cfg::kVOff) + st * Cfg::kKTileBytes;
                    tc::mbar_arrive_expect_tx_warp(bar, static_cast<uint32_t>(nvalid) * bs * DQ * 2);
                    for (int b = 0; b < per_tile; ++b) {
                        const int blk = __shfl_sync(0xffffffffu, blk_cur, b);
                        if (b < nvalid) {
#pragma unroll
                            for (int h = 0; h < DQ / 64; ++h)
                                tc::tma_load_4d_warp(dst + h * Cfg::kHalf + b * bs * 128, map, bar, h * 64, ukvh, 0, blk);
                        }
                    }
                } else {
                    const uint32_t dst = s_base + (is_k ? st * Cfg::kKTileBytes : Cfg::kVOff + st * Cfg::kVTileBytes);
                    const int dcols = is_k ? DQ : DV;
                    tc::mbar_arrive_expect_tx_warp(bar, static_cast<uint32_t>(nvalid) * bs * dcols * 2);
                    for (int b = 0; b < per_tile; ++b) {
                        const int blk = __shfl_sync(0xffffffffu, blk_cur, b);
                        if (b < nvalid) {
                            if (is_k) {
#pragma unroll
                                for (int h = 0; h < DQ / 64; ++h)
                                    tc::tma_load_4d_warp(dst + h * Cfg::kHalf + b * bs * 128, map, bar, h * 64, ukvh, 0, blk);
                            } else {
#pragma unroll
                                for (int h = 0; h < DV / 64; ++h)
                                    tc::tma_load_4d_warp(dst + h * Cfg::kHalf + b * bs * 128, map, bar, h * 64, ukvh, 0, blk);
                            }
                        }
                    }
                }
                if (!is_k && i == it.ntiles - 1 && it.tail_fix) {
                    // zero V rows of keys >= ctx (stale slots, unloaded blocks)
                    if (!wait(VFULL(st), (g / nst) & 1)) { ok = false; break; }
                    const int r0 = it.ctx - (it.kt0 + i) * kKeys;
                    const int nrows = kKeys - r0;
                    for (int e = lane; e < nrows * 8 * (DV / 64); e += 32) {
                        const int h = e / (nrows * 8), rem = e % (nrows * 8);
                        const int row = r0 + rem / 8, ch = rem % 8;
                        *reinterpret_cast<uint4 *>(smem + Cfg::kVOff + st * Cfg::kVTileBytes + h * Cfg::kHalf +
                                                   row * 128 + ch * 16) = make_uint4(0u, 0u, 0u, 0u);
                    }
                    tc::fence_proxy_async_smem();
                    __syncwarp();
                    tc::mbar_arrive_warp(VZERO);
                    ++nfix;
                }
            }
            if (!ok) break;
            if (!is_k) tc::mbar_arrive_warp(ITEMEMPTY(slot));
        }
    } else if (warp == 10) {
        // -------------------------------------------------------- MMA issuer
        // The loop runs with warp-uniform values (passed through __shfl_sync
        // so the compiler keeps them in uniform registers); each tcgen05
        // instruction is issued by one elected lane.
        constexpr uint32_t idS = F16 ? tc::idesc_f16(kRows, kKeys, false) : tc::idesc_bf16(kRows, kKeys, false);
        constexpr uint32_t idO = F16 ? tc::idesc_f16(kRows, DV, true) : tc::idesc_bf16(kRows, DV, true);
        const uint32_t utmem = __shfl_sync(0xffffffffu, tmem, 0);
        const uint32_t us_base = __shfl_sync(0xffffffffu, s_base, 0);
        int gk = 0, gv = 0, t = 0, nfix = 0;
        bool ok = true, issued = false;
        auto issue_s = [&](int w, int st_in) {
            const int st = __shfl_sync(0xffffffffu, st_in, 0);
            const uint64_t kd = tc::sdesc_sw128(us_base + st * Cfg::kKTileBytes, 16, 1024);
            const uint64_t qd = tc::sdesc_sw128(us_base + Cfg::kQOff + w * Cfg::kQBytes, 16, 1024);
            const uint32_t dS = utmem + col_s(w);
#pragma unroll
            for (int kk = 0; kk < DQ / 16; ++kk)
                tc::mma_ss_warp(dS, qd + ((kk / 4) * Cfg::kQHalf + (kk % 4) * 32) / 16,
                                kd + ((kk / 4) * Cfg::kHalf + (kk % 4) * 32) / 16, idS, kk > 0);
            tc::commit_warp(SFULL(w));
            issued = true;
        };
        auto issue_pv = [&](int w, int st_in, uint32_t acc_in) {
            const int st = __shfl_sync(0xffffffffu, st_in, 0);
            const uint32_t acc = __shfl_sync(0xffffffffu, acc_in, 0);
            const uint64_t vd =
                tc::sdesc_sw128(us_base + Cfg::kVOff + st * Cfg::kVTileBytes, Cfg::kHalf, 1024);
            const uint32_t dO = utmem + col_o(w), aP = utmem + col_s(w);
            tc::mma_ts_warp(dO, aP, vd, idO, acc);
#pragma unroll
            for (int kk = 1; kk < kKeys / 16; ++kk) tc::mma_ts_warp(dO, aP + kk * 8, vd + (kk * 2048) / 16, idO, 1u);
            issued = true;
        };
        for (int k = 0; ok; ++k) {
            const int slot = k & 1;
            if (!wait(ITEMFULL(slot), (k >> 1) & 1)) { ok = false; break; }
            const int idx = __shfl_sync(0xffffffffu, item_slot[slot], 0);
            if (idx < 0) break;
            const ItemGeom it = item_geom(p, idx);
            const int n = __shfl_sync(0xffffffffu, it.ntiles, 0);
            const bool tail = __shfl_sync(0xffffffffu, it.tail_fix ? 1 : 0, 0) != 0;
            // S_0(0), S_1(0)
            if (!wait(QFULL, k & 1)) { ok = false; break; }
            if (!wait(KFULL(gk % kKStages), (gk / kKStages) & 1)) { ok = false; break; }
            tc::fence_after_sync();
            issue_s(0, gk % kKStages);
            issue_s(1, gk % kKStages);
            tc::commit_warp(KEMPTY(gk % kKStages));
            ++gk;
            if (n == 1) tc::commit_warp(QEMPTY);
            for (int j = 0; j < n; ++j) {
                const int T = t + j, vst = gv % kVStages;
                if (j == n - 1 && tail) {
                    if (!wait(VZERO, nfix & 1)) { ok = false; break; }
                } else if (!wait(VFULL(vst), (gv / kVStages) & 1)) {
                    ok = false;
                    break;
                }
                // O_0 += P_0(j) V(j), then S_0(j + 1)
                if (!wait(PFULL(0), T & 1)) { ok = false; break; }
                if (j == 0 && k >= 1 && !wait(OFREE(0), (k - 1) & 1)) { ok = false; break; }
                tc::fence_after_sync();
                issue_pv(0, vst, j > 0 ? 1u : 0u);
                if (j == n - 1) tc::commit_warp(ODONE(0));
                const bool more = j + 1 < n;
                // (one V stage: both P V first, so that the next V tile loads
                // while both S of the next key tile run)
                constexpr bool kPvFirst = Cfg::kVStages == 1;
                if (!kPvFirst && more) {
                    if (!wait(KFULL(gk % kKStages), (gk / kKStages) & 1)) { ok = false; break; }
                    tc::fence_after_sync();
                    issue_s(0, gk % kKStages);
                }
                // O_1 += P_1(j) V(j), then S_1(j + 1)
                if (!wait(PFULL(1), T & 1)) { ok = false; break; }
                if (j == 0 && k >= 1 && !wait(OFREE(1), (k - 1) & 1)) { ok = false; break; }
                tc::fence_after_sync();
                issue_pv(1, vst, j > 0 ? 1u : 0u);
                tc::commit_warp(VEMPTY(vst));
                ++gv;
                if (j == n - 1) tc::commit_warp(ODONE(1));
                if (kPvFirst && more) {
                    if (!wait(KFULL(gk % kKStages), (gk / kKStages) & 1)) { ok = false; break; }
                    tc::fence_after_sync();
                    issue_s(0, gk % kKStages);
                }
                if (more) {
                    issue_s(1, gk % kKStages);
                    tc::commit_warp(KEMPTY(gk % kKStages));
                    ++gk;
                    if (j + 1 == n - 1) tc::commit_warp(QEMPTY);  // last S of this item
                }
            }
            if (!ok) break;
            t += n;
            if (tail) ++nfix;
            tc::mbar_arrive_warp(ITEMEMPTY(slot));
        }
        if (!ok && issued) {  // drain whatever is still in flight
            tc::commit_warp(DRAIN);
            tc::mbar_wait(DRAIN, 0, 200000000ull);
        }
    }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;\n" ::"n"(kRegsSoftmax));
        // ------------------------------------------- softmax / epilogue rows
        const int w = warp >> 2;                 // warpgroup = Q tile
        const int r = tid & 127;                 // MMA row = TMEM lane
        const uint32_t lane_addr = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
        const int pl = r / G, hl = r % G;
        const float sc = p.scale_log2;
        int t = 0;
        for (int k = 0;; ++k) {
            const int slot = k & 1;
            if (!wait(ITEMFULL(slot), (k >> 1) & 1)) break;
            const int idx = item_slot[slot];
            if (idx < 0) break;
            const ItemGeom it = item_geom(p, idx);
            const int pw = it.p0 + w * P;
            const bool row_ok = (r < P * G) && (pw + pl < it.p0 + it.rows);
            // rows past the item (padding) keep a position too; their results are
            // never stored, so they need no masking of their own
            const int pos = it.prefix + pw + pl;
            const int min_pos = it.prefix + pw;
            const int64_t tok = it.q_start + pw + pl;
            const int head = it.kvh * G + hl;

            float m_run = -INFINITY;  // reference max (log2 units) of the exponentials
            float l = 0.f;
            bool ok = true;
            for (int i = 0; i < it.ntiles; ++i) {
                const int T = t + i;
                if (!wait(SFULL(w), T & 1)) { ok = false; break; }
                tc::fence_after_sync();
                uint32_t s[kKeys];
#pragma unroll
                for (int c = 0; c < kKeys / 32; ++c)
                    tc::tmem_ld32(lane_addr + col_s(w) + 32 * c, *reinterpret_cast<uint32_t(*)[32]>(&s[32 * c]));
                tc::tmem_wait_ld();
                // tiles that reach past the first row's position need the causal
                // mask; all others are fully visible to every row of the tile
                const int k0 = (it.kt0 + i) * kKeys;
                const bool masked_tile = k0 + kKeys - 1 > min_pos;
                if (masked_tile) {
#pragma unroll
                    for (int j = 0; j < kKeys; ++j)
                        if (k0 + j > pos) s[j] = __float_as_uint(-INFINITY);
                }
                float mx0 = -INFINITY, mx1 = -INFINITY, mx2 = -INFINITY, mx3 = -INFINITY;
#pragma unroll
                for (int j = 0; j < kKeys; j += 8) {
                    mx0 = fmax3(mx0, __uint_as_float(s[j]), __uint_as_float(s[j + 1]));
                    mx1 = fmax3(mx1, __uint_as_float(s[j + 2]), __uint_as_float(s[j + 3]));
                    mx2 = fmax3(mx2, __uint_as_float(s[j + 4]), __uint_as_float(s[j + 5]));
                    mx3 = fmax3(mx3, __uint_as_float(s[j + 6]), __uint_as_float(s[j + 7]));
                }
                // the scale is positive, so the max of scaled scores is the scaled max
                const float tmax = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * sc;
                const bool need = (m_run == -INFINITY) ? (tmax != -INFINITY) : (tmax > m_run + kRescaleThreshold);
                if (__any_sync(0xffffffffu, need)) {
                    const float m_new = need ? fmaxf(m_run, tmax) : m_run;
                    const float alpha = (need && m_run != -INFINITY) ? fast_exp2(m_run - m_new) : 1.f;
                    if (i > 0) {
                        // PV_w(i - 1) is complete: S_w(i) was issued after it
#pragma unroll
                        for (int c = 0; c < DV / 32; ++c) {
                            uint32_t o[32];
                            tc::tmem_ld32(lane_addr + col_o(w) + 32 * c, o);
                            tc::tmem_wait_ld();
#pragma unroll
                            for (int j = 0; j < 32; ++j) o[j] = __float_as_uint(__uint_as_float(o[j]) * alpha);
                            tc::tmem_st32(lane_addr + col_o(w) + 32 * c, o);
                        }
                    }
                    l *= alpha;
                    m_run = m_new;
                }
                const float nbase = (m_run == -INFINITY) ? 0.f : -m_run;
                // x = s * scale - m and the row sum on paired fp32 lanes
                const uint64_t sc2 = f2_pack(sc, sc), nb2 = f2_pack(nbase, nbase);
                uint64_t lacc0 = f2_pack(0.f, 0.f), lacc1 = lacc0;
#pragma unroll
                for (int q4 = 0; q4 < kKeys / 32; ++q4) {
                    uint32_t pk[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const uint64_t x2 = f2_fma(f2_pack(__uint_as_float(s[32 * q4 + 2 * j]),
                                                           __uint_as_float(s[32 * q4 + 2 * j + 1])), sc2, nb2);
                        float x0, x1;
                        f2_unpack(x2, x0, x1);
                        const float p0 = fast_exp2(x0), p1 = fast_exp2(x1);
                        if (j & 1) lacc1 = f2_add(lacc1, f2_pack(p0, p1));
                        else lacc0 = f2_add(lacc0, f2_pack(p0, p1));
                        pk[j] = F16 ? pack_f16x2(p0, p1) : pack_bf16x2(p0, p1);
                    }
                    tc::tmem_st16(lane_addr + col_s(w) + 16 * q4, pk);
                }
                {
                    float a0, a1;
                    f2_unpack(f2_add(lacc0, lacc1), a0, a1);
                    l += a0 + a1;
                }
                tc::tmem_wait_st();
                tc::fence_before_sync();
                tc::mbar_arrive(PFULL(w));
            }
            if (!ok) break;
            if (!wait(ODONE(w), k & 1)) break;
            tc::fence_after_sync();
            const float inv = 1.f / l;
            uint4 *orow = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(p.out) +
                                                    (tok * p.num_q_heads + head) * DV);
            if (it.ns == 1) {
#pragma unroll
                for (int c = 0; c < DV / 32; ++c) {
                    uint32_t o[32];
                    tc::tmem_ld32(lane_addr + col_o(w) + 32 * c, o);
                    tc::tmem_wait_ld();
                    if (row_ok) {
                        // 32-byte stores: whole sectors of this row
#pragma unroll
                        for (int j = 0; j < 2; ++j) {
                            uint32_t v[8];
#pragma unroll
                            for (int x = 0; x < 8; ++x)
                                v[x] = pack_bf16x2(__uint_as_float(o[16 * j + 2 * x]) * inv,
                                                   __uint_as_float(o[16 * j + 2 * x + 1]) * inv);
                            st_global_v8(orow + c * 4 + 2 * j, v[0], v[1], v[2], v[3], v[4], v[5], v[6], v[7]);
                        }
                    }
                }
                if (row_ok) p.lse[tok * p.num_q_heads + head] = (m_run + log2f(l)) * kLn2;
            } else {
                // a key split: store O / l and m + log2 l of this split (the
                // partial of Eq. 1 over its keys), row r of the tile at float4
                // column q in position q * 128 + r, so that a warp's stores
                // and loads are contiguous
                const int64_t prow = (static_cast<int64_t>(it.pbase + it.split) * 2 + w) * 128;
                float4 *po = reinterpret_cast<float4 *>(p.ppart_o) + prow * (DV / 4) + r;
#pragma unroll
                for (int c = 0; c < DV / 32; ++c) {
                    uint32_t o[32];
                    tc::tmem_ld32(lane_addr + col_o(w) + 32 * c, o);
                    tc::tmem_wait_ld();
#pragma unroll
                    for (int j = 0; j < 8; ++j)
                        po[(c * 8 + j) * 128] = make_float4(__uint_as_float(o[4 * j]) * inv, __uint_as_float(o[4 * j + 1]) * inv,
                                                            __uint_as_float(o[4 * j + 2]) * inv, __uint_as_float(o[4 * j + 3]) * inv);
                }
                const float my_lse = m_run + log2f(l);
                p.ppart_lse[prow + r] = my_lse;
                // the last split of this tile pair to finish merges, warp by warp
                __threadfence();
                __syncwarp();
                int last = 0;
                if (lane == 0) last = atomicAdd(p.pcounters + it.cnt * 8 + (warp & 7), 1) == it.ns - 1;
                last = __shfl_sync(0xffffffffu, last, 0);
                if (last) {
                    __threadfence();
                    auto lse_of = [&](int sp) {
                        return __ldcg(p.ppart_lse + (static_cast<int64_t>(it.pbase + sp) * 2 + w) * 128 + r);
                    };
                    // sums run in split order, whichever split merges, so
                    // that a run is reproducible bit for bit
                    float M = -INFINITY;
                    for (int sp = 0; sp < it.ns; ++sp) M = fmaxf(M, sp == it.split ? my_lse : lse_of(sp));
                    float L = 0.f;
                    for (int sp = 0; sp < it.ns; ++sp) L += fast_exp2((sp == it.split ? my_lse : lse_of(sp)) - M);
                    const float iL = 1.f / L;
#pragma unroll 1
                    for (int c = 0; c < DV / 32; ++c) {
                        uint32_t o[32];
                        tc::tmem_ld32(lane_addr + col_o(w) + 32 * c, o);
                        tc::tmem_wait_ld();
                        float4 acc[8];
#pragma unroll
                        for (int j = 0; j < 8; ++j) acc[j] = make_float4(0.f, 0.f, 0.f, 0.f);
                        for (int sp = 0; sp < it.ns; ++sp) {
                            float4 v[8];
                            float ws;
                            if (sp == it.split) {
                                ws = fast_exp2(my_lse - M);
#pragma unroll
                                for (int j = 0; j < 8; ++j)
                                    v[j] = make_float4(__uint_as_float(o[4 * j]) * inv, __uint_as_float(o[4 * j + 1]) * inv,
                                                       __uint_as_float(o[4 * j + 2]) * inv, __uint_as_float(o[4 * j + 3]) * inv);
                            } else {
                                ws = fast_exp2(lse_of(sp) - M);
                                const float4 *q4 = reinterpret_cast<const float4 *>(p.ppart_o) +
                                                   (static_cast<int64_t>(it.pbase + sp) * 2 + w) * 128 * (DV / 4) + r;
#pragma unroll
                                for (int j = 0; j < 8; ++j) v[j] = __ldcg(q4 + (c * 8 + j) * 128);
                            }
#pragma unroll
                            for (int j = 0; j < 8; ++j) {
                                acc[j].x += ws * v[j].x; acc[j].y += ws * v[j].y;
                                acc[j].z += ws * v[j].z; acc[j].w += ws * v[j].w;
                            }
                        }
                        if (row_ok) {
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                uint4 v;
                                v.x = pack_bf16x2(acc[2 * j].x * iL, acc[2 * j].y * iL);
                                v.y = pack_bf16x2(acc[2 * j].z * iL, acc[2 * j].w * iL);
                                v.z = pack_bf16x2(acc[2 * j + 1].x * iL, acc[2 * j + 1].y * iL);
                                v.w = pack_bf16x2(acc[2 * j + 1].z * iL, acc[2 * j + 1].w * iL);
                                orow[c * 4 + j] = v;
                            }
                        }
                    }
                    if (row_ok) p.lse[tok * p.num_q_heads + head] = (M + log2f(L)) * kLn2;
                    if (lane == 0) p.pcounters[it.cnt * 8 + (warp & 7)] = 0;  // ready for the next run
                }
            }
            t += it.ntiles;
            tc::fence_before_sync();
            tc::mbar_arrive(OFREE(w));  // O_w may be overwritten by the next item
            tc::mbar_arrive(ITEMEMPTY(slot));
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, kTmemCols);
    }
    if (tid == 0) {  // the last CTA out resets the work queue (and the append count) for the next run
        __threadfence();
        if (atomicAdd(p.sched + 1, 1) == static_cast<int>(gridDim.x) - 1) {
            p.sched[0] = 0;
            p.sched[1] = 0;
            if (p.fa_count != nullptr) *p.fa_count = 0;
            __threadfence();
        }
    }
}

// 4-D map over a paged cache [num_blocks, bs, Hkv, d]: box = one block of one
// kv head, 64 columns wide, 128-byte swizzle.
bool encode_cache_map(CUtensorMap *m, const void *base, int d, int hkv, int bs, int nblocks, bool f16) {
    EncodeTiledFn enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(hkv), static_cast<cuuint64_t>(bs),
                          static_cast<cuuint64_t>(nblocks)};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(d) * 2, static_cast<cuuint64_t>(hkv) * d * 2,
                             static_cast<cuuint64_t>(bs) * hkv * d * 2};
    cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(bs), 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return enc(m, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base),
               dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D map over q [T, Hq, d]: box = 64 columns x G heads x P positions, so a
// box lands as the packed (position, head) rows of one Q tile.
bool encode_q_map(CUtensorMap *m, const void *base, int d, int hq, int64_t T, int G, int P, bool f16) {
    EncodeTiledFn enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(hq), static_cast<cuuint64_t>(T)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(d) * 2, static_cast<cuuint64_t>(hq) * d * 2};
    cuuint32_t box[3] = {64, static_cast<cuuint32_t>(G), static_cast<cuuint32_t>(P)};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base),
               dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DQ, int DV, bool F16>
int launch_tc(const AttnParams &p, cudaStream_t st, int max_ctas, cudaEvent_t started, bool pdl) {
    using Cfg = TcCfg<DQ, DV>;
    TcMaps maps;
    if (!encode_cache_map(&maps.k, p.k_cache, DQ, p.num_kv_heads, p.block_size, p.num_blocks, F16) ||
        !encode_cache_map(&maps.v, p.v_cache, DV, p.num_kv_heads, p.block_size, p.num_blocks, F16) ||
        !encode_q_map(&maps.q, p.q, DQ, p.num_q_heads, p.num_tokens, p.group, kRows / p.group, F16))
        return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled");
    auto kernel = prefill_tc_kernel<DQ, DV, F16>;
    FNPU_CUDA_TRY(cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes));
    FNPU_CUDA_TRY(cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                       cudaSharedmemCarveoutMaxShared));
    const int grid = p.num_pitems < max_ctas ? p.num_pitems : max_ctas;
    FNPU_CUDA_TRY(launch_coop(kernel, grid, kThreads, Cfg::kSmemBytes, st, pdl, started, p.fa_count != nullptr, p,
                              maps));
    return FNPU_OK;
}

}  // namespace

bool prefill_tc_supported(int d_qk, int d_v, int block_size, int group) {
    // split K/V heads of 64 or 128; the per-head keys (192) and values (128)
    // of an expanded latent cache, one kv head per query head
    const bool dims = (d_qk == d_v && (d_qk == 64 || d_qk == 128)) || (d_qk == 192 && d_v == 128 && group == 1);
    return dims && (block_size == 16 || block_size == 32 || block_size == 64) && group >= 1 && group <= kRows;
}

// positions per work item: two Q tiles of floor(128 / G) positions each
int prefill_tc_rows_per_item(int group) { return 2 * (kRows / group); }

// keys per K/V tile (the unit of the planner's key splits)
int prefill_tc_keys_per_tile() { return kKeys; }

int launch_prefill_tc(const AttnParams &p, void *stream, int max_ctas, void *started, bool f16, bool pdl) {
    if (p.num_pitems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaEvent_t ev = static_cast<cudaEvent_t>(started);
    if (f16)
        return p.head_dim_qk == 128 && p.head_dim_v == 128 ? launch_tc<128, 128, true>(p, st, max_ctas, ev, pdl)
                                                            : FNPU_EUNSUPPORTED;
    if (p.head_dim_qk == 64 && p.head_dim_v == 64) return launch_tc<64, 64, false>(p, st, max_ctas, ev, pdl);
    if (p.head_dim_qk == 128 && p.head_dim_v == 128)
        return launch_tc<128, 128, false>(p, st, max_ctas, ev, pdl);
    if (p.head_dim_qk == 192 && p.head_dim_v == 128)
        return launch_tc<192, 128, false>(p, st, max_ctas, ev, pdl);
    return FNPU_EUNSUPPORTED;
}

}  // namespace fnpu
