// Decode split-KV attention for callers that cannot allocate device memory.
//
// Some callers are not allowed to call cudaMalloc at all: code that runs
// inside another framework's memory pool or a pre-reserved arena, a driver of
// a fixed-memory serving process, or any code that must not add device
// allocations of its own. The regular path needs a plan, and a plan owns a
// cudaMalloc'd workspace (work list, split scratch). This entry point is the
// same GQA-packed split-KV decode computation, with its split scratch in one
// fixed array in the library's own device memory instead:
//
//   * the work list is implicit: CTA b handles split b % max_splits of
//     (sequence, kv head) b / max_splits, reading the context length on the
//     device, so nothing is planned or uploaded;
//   * partial outputs, partial log-sum-exps and the merge counters live in
//     g_noalloc_scratch (FNPU_NOALLOC_SCRATCH_BYTES, defined below), which
//     every GPU that loads this library holds from load until the process
//     exits; requests that need more are rejected;
//   * the counters are cleared with cudaMemsetAsync at the start of every
//     call (it allocates nothing);
//   * the context lengths and block ids are only seen on the device, so the
//     kernel checks them there: a context outside [1, max_context_len] is
//     skipped, and a block id outside [0, num_blocks) is never loaded; both
//     raise the library-wide device error flag (fnpu_check reports it), and
//     no load leaves the caller's block-table rows or pools.
//
// The host code cannot pass g_noalloc_scratch itself to a kernel: in host code
// that name is a host-side shadow, not a device address. The device address
// is looked up once per device with cudaGetSymbolAddress while that device is
// current, during the first call made on it.
#include <math.h>

#include <mutex>

#include "common.cuh"

namespace fnpu {
namespace {

constexpr int kThreads = 128;
constexpr int kTileKeys = 64;
constexpr int kStages = 3;
constexpr int kMaxDevices = 64;
constexpr size_t kScratchFloats = FNPU_NOALLOC_SCRATCH_BYTES / sizeof(float);

__device__ __align__(256) float g_noalloc_scratch[kScratchFloats];

struct NoallocParams {
    const __nv_bfloat16 *q;  // [num_seqs, Hq, D]
    const __nv_bfloat16 *k_cache, *v_cache;
    __nv_bfloat16 *out;      // [num_seqs, Hq, D]
    float *lse;              // [num_seqs, Hq]
    const int32_t *context_len;
    const int32_t *block_table;
    int32_t bt_stride, num_q_heads, num_kv_heads, group, block_size;
    int32_t max_splits, split_keys;
    int32_t max_context_len, num_blocks;  // the host's bounds, checked on the device
    int32_t *err;                         // library-wide device error flag (bit 1)
    int64_t k_slot_stride, v_slot_stride;
    float scale_log2;
    int32_t *counters;  // [num_seqs * Hkv] inside the scratch
    float *part_lse;    // [num_seqs * Hkv * max_splits, group]
    float *part_o;      // [num_seqs * Hkv * max_splits, group, D]
};

__device__ __forceinline__ uint32_t swz_off(int row, int chunk, int row_bytes) {
    return static_cast<uint32_t>(row * row_bytes + ((chunk ^ (row & 7)) << 4));
}

template <int D>
__global__ void __launch_bounds__(kThreads, 2) decode_noalloc_kernel(const NoallocParams p) {
    constexpr int kChunks = D / 8;
    constexpr int kTileBytes = kTileKeys * D * 2;
    constexpr int kStageBytes = 2 * kTileBytes;
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int s_last;

    const int split = blockIdx.x % p.max_splits;
    const int grp = blockIdx.x / p.max_splits;
    const int kvh = grp % p.num_kv_heads;
    const int seq = grp / p.num_kv_heads;
    const int ctx = p.context_len[seq];
    if (ctx < 1 || ctx > p.max_context_len) {
        // the host's bound sized the grid and the block-table rows: such a
        // sequence is skipped (its out and lse rows are left as they were)
        if (split == 0 && threadIdx.x == 0) atomicOr(p.err, 2);
        return;
    }
    // ctx <= max_context_len, so nsp <= max_splits and every key's block-table
    // entry lies inside the row (stride >= ceil(max_context_len / bs))
    const int nsp = (ctx + p.split_keys - 1) / p.split_keys;
    if (split >= nsp) return;
    const int key_begin = split * p.split_keys;
    const int key_end = (split == nsp - 1) ? ctx : key_begin + p.split_keys;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, c = lane & 3;
    const int G = p.group;
    const __nv_bfloat16 *qrow = p.q + (static_cast<int64_t>(seq) * p.num_q_heads + kvh * G) * D;
    uint32_t qb[D / 16][2];
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
        if (g < G) {
            qb[kk][0] = *reinterpret_cast<const uint32_t *>(qrow + g * D + kk * 16 + 2 * c);
            qb[kk][1] = *reinterpret_cast<const uint32_t *>(qrow + g * D + kk * 16 + 8 + 2 * c);
        } else {
            qb[kk][0] = qb[kk][1] = 0u;
        }
    }

    const int nkeys = key_end - key_begin;
    const int ntiles = (nkeys + kTileKeys - 1) / kTileKeys;
    const int32_t *bt = p.block_table + static_cast<int64_t>(seq) * p.bt_stride;
    const int bs = p.block_size;
    const uint32_t smem_base = smem_u32(smem);
    auto load_tile = [&](int tile, int stage) {
        const uint32_t sK = smem_base + stage * kStageBytes;
        const uint32_t sV = sK + kTileBytes;
        const int kb = key_begin + tile * kTileKeys;
#pragma unroll 4
        for (int i = tid; i < kTileKeys * kChunks; i += kThreads) {
            const int row = i / kChunks, ch = i % kChunks;
            const int key = kb + row;
            bool valid = key < key_end;
            int64_t slot = 0;
            if (valid) {
                const int blk = __ldg(bt + key / bs);
                if (blk < 0 || blk >= p.num_blocks) {
                    // never loaded (the stage is zero-filled); the result of
                    // this sequence is undefined and the flag says so
                    valid = false;
                    if (ch == 0) atomicOr(p.err, 2);
                } else {
                    slot = static_cast<int64_t>(blk) * bs + key % bs;
                }
            }
            const uint32_t off = swz_off(row, ch, D * 2);
            cp_async_16(sK + off, p.k_cache + slot * p.k_slot_stride + kvh * D + ch * 8, valid);
            cp_async_16(sV + off, p.v_cache + slot * p.v_slot_stride + kvh * D + ch * 8, valid);
        }
    };

    float o[D / 16][4];
#pragma unroll
    for (int mt = 0; mt < D / 16; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
#pragma unroll
    for (int s = 0; s < kStages - 1; ++s) {
        if (s < ntiles) load_tile(s, s);
        cp_async_commit();
    }
    const int lj = lane >> 3, lr = lane & 7;
    for (int tile = 0; tile < ntiles; ++tile) {
        const int pre = tile + kStages - 1;
        if (pre < ntiles) load_tile(pre, pre % kStages);
        cp_async_commit();
        cp_async_wait<kStages - 1>();
        __syncthreads();
        const uint32_t sK = smem_base + (tile % kStages) * kStageBytes;
        const uint32_t sV = sK + kTileBytes;
        float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
            uint32_t a0, a1, a2, a3;
            const int row = 16 * warp + lr + 8 * (lj & 1);
            ldmatrix_x4(a0, a1, a2, a3, sK + swz_off(row, 2 * kk + (lj >> 1), D * 2));
            mma_bf16_16816(s, a0, a1, a2, a3, qb[kk][0], qb[kk][1]);
        }
        const int kr = tile * kTileKeys + 16 * warp + g;
        const bool v0 = kr < nkeys, v1 = kr + 8 < nkeys;
        const float x0 = v0 ? s[0] * p.scale_log2 : -INFINITY;
        const float x1 = v0 ? s[1] * p.scale_log2 : -INFINITY;
        const float x2 = v1 ? s[2] * p.scale_log2 : -INFINITY;
        const float x3 = v1 ? s[3] * p.scale_log2 : -INFINITY;
        float t0 = fmaxf(x0, x2), t1 = fmaxf(x1, x3);
        t0 = warp_max_xor(t0, 4); t0 = warp_max_xor(t0, 8); t0 = warp_max_xor(t0, 16);
        t1 = warp_max_xor(t1, 4); t1 = warp_max_xor(t1, 8); t1 = warp_max_xor(t1, 16);
        const float mn0 = fmaxf(m0, t0), mn1 = fmaxf(m1, t1);
        const float b0 = (mn0 == -INFINITY) ? 0.f : mn0;
        const float b1 = (mn1 == -INFINITY) ? 0.f : mn1;
        const float al0 = fast_exp2(m0 - b0), al1 = fast_exp2(m1 - b1);
        const float p0 = fast_exp2(x0 - b0), p1 = fast_exp2(x1 - b1);
        const float p2 = fast_exp2(x2 - b0), p3 = fast_exp2(x3 - b1);
        l0 = l0 * al0 + p0 + p2;
        l1 = l1 * al1 + p1 + p3;
        m0 = mn0;
        m1 = mn1;
#pragma unroll
        for (int mt = 0; mt < D / 16; ++mt) {
            o[mt][0] *= al0; o[mt][1] *= al1; o[mt][2] *= al0; o[mt][3] *= al1;
        }
        const uint32_t pb0 = movmatrix_trans(pack_bf16x2(p0, p1));
        const uint32_t pb1 = movmatrix_trans(pack_bf16x2(p2, p3));
#pragma unroll
        for (int mt = 0; mt < D / 16; ++mt) {
            uint32_t a0, a1, a2, a3;
            const int row = 16 * warp + lr + 8 * (lj >> 1);
            ldmatrix_x4_trans(a0, a1, a2, a3, sV + swz_off(row, 2 * mt + (lj & 1), D * 2));
            mma_bf16_16816(o[mt], a0, a1, a2, a3, pb0, pb1);
        }
        __syncthreads();
    }
    cp_async_wait<0>();
    l0 += __shfl_xor_sync(0xffffffffu, l0, 4);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 8);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 16);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 4);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 8);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 16);

    __syncthreads();
    float *sm_ml = reinterpret_cast<float *>(smem);
    float *sm_o = sm_ml + 4 * 8 * 2;
    if (g == 0) {
        sm_ml[(warp * 8 + 2 * c) * 2 + 0] = m0;
        sm_ml[(warp * 8 + 2 * c) * 2 + 1] = l0;
        sm_ml[(warp * 8 + 2 * c + 1) * 2 + 0] = m1;
        sm_ml[(warp * 8 + 2 * c + 1) * 2 + 1] = l1;
    }
#pragma unroll
    for (int mt = 0; mt < D / 16; ++mt) {
        float *w0 = sm_o + (warp * 8 + 2 * c) * D + mt * 16 + g;
        float *w1 = sm_o + (warp * 8 + 2 * c + 1) * D + mt * 16 + g;
        w0[0] = o[mt][0];
        w1[0] = o[mt][1];
        w0[8] = o[mt][2];
        w1[8] = o[mt][3];
    }
    __syncthreads();

    const int64_t part = static_cast<int64_t>(grp) * p.max_splits + split;
    for (int idx = tid; idx < G * D; idx += kThreads) {
        const int h = idx / D, d = idx % D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < 4; ++w) M = fmaxf(M, sm_ml[(w * 8 + h) * 2]);
        float L = 0.f, acc = 0.f;
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const float mw = sm_ml[(w * 8 + h) * 2];
            const float sc = (mw == -INFINITY) ? 0.f : fast_exp2(mw - M);
            L += sc * sm_ml[(w * 8 + h) * 2 + 1];
            acc += sc * sm_o[(w * 8 + h) * D + d];
        }
        const float lse2 = M + log2f(L);
        const int qh = kvh * G + h;
        if (nsp == 1) {
            p.out[(static_cast<int64_t>(seq) * p.num_q_heads + qh) * D + d] = __float2bfloat16_rn(acc / L);
            if (d == 0) p.lse[static_cast<int64_t>(seq) * p.num_q_heads + qh] = lse2 * kLn2;
        } else {
            p.part_o[(part * G + h) * D + d] = acc / L;
            if (d == 0) p.part_lse[part * G + h] = lse2;
        }
    }
    if (nsp == 1) return;

    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = (atomicAdd(p.counters + grp, 1) == nsp - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    const int64_t base = static_cast<int64_t>(grp) * p.max_splits;
    for (int idx = tid; idx < G * D; idx += kThreads) {
        const int h = idx / D, d = idx % D;
        float M = -INFINITY;
        for (int sp = 0; sp < nsp; ++sp) M = fmaxf(M, __ldcg(p.part_lse + (base + sp) * G + h));
        float L = 0.f, acc = 0.f;
        for (int sp = 0; sp < nsp; ++sp) {
            const float w = fast_exp2(__ldcg(p.part_lse + (base + sp) * G + h) - M);
            L += w;
            acc += w * __ldcg(p.part_o + ((base + sp) * G + h) * D + d);
        }
        const int qh = kvh * G + h;
        p.out[(static_cast<int64_t>(seq) * p.num_q_heads + qh) * D + d] = __float2bfloat16_rn(acc / L);
        if (d == 0) p.lse[static_cast<int64_t>(seq) * p.num_q_heads + qh] = (M + log2f(L)) * kLn2;
    }
    if (tid == 0) p.counters[grp] = 0;
}

std::mutex g_setup_mu;
float *g_scratch_addr[kMaxDevices] = {};

// Device address of g_noalloc_scratch on the current device, looked up once
// per device (the first call on a device does it; see fnpu.h).
int scratch_address(float **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return FNPU_ECUDA;
    if (dev < 0 || dev >= kMaxDevices) return FNPU_EUNSUPPORTED;
    std::lock_guard<std::mutex> lk(g_setup_mu);
    if (!g_scratch_addr[dev]) {
        void *ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) {
            cudaGetLastError();
            return FNPU_ECUDA;
        }
        g_scratch_addr[dev] = static_cast<float *>(ptr);
    }
    *out = g_scratch_addr[dev];
    return FNPU_OK;
}

template <int D>
int launch_noalloc(const NoallocParams &p, int grid, cudaStream_t st) {
    constexpr int kSmem = kStages * 2 * kTileKeys * D * 2;
    if (cudaFuncSetAttribute(decode_noalloc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kSmem) != cudaSuccess)
        return FNPU_ECUDA;
    decode_noalloc_kernel<D><<<grid, kThreads, kSmem, st>>>(p);
    return cudaGetLastError() == cudaSuccess ? FNPU_OK : FNPU_ECUDA;
}

}  // namespace
}  // namespace fnpu

using namespace fnpu;

extern "C" int fnpu_decode_attn_noalloc(const fnpu_attn_desc *desc, int32_t num_seqs,
                                        const int32_t *context_len, const int32_t *block_table,
                                        int32_t block_table_stride, int32_t max_context_len,
                                        int32_t split_keys, const void *q, const void *k_cache,
                                        const void *v_cache, void *out, float *lse, void *stream) {
    if (!desc || num_seqs < 0) return FNPU_EINVAL;
    const int32_t Hq = desc->num_q_heads, Hkv = desc->num_kv_heads, D = desc->head_dim_qk;
    if (Hq <= 0 || Hkv <= 0 || Hq % Hkv || desc->block_size <= 0 || desc->num_blocks <= 0)
        return FNPU_EINVAL;
    if (desc->kv_fp8 != 0 && desc->kv_fp8 != 1) return FNPU_EINVAL;
    if (desc->v_in_k_latent || desc->kv_fp8 || desc->head_dim_v != D || (D != 64 && D != 128) || Hq / Hkv > 8)
        return FNPU_EUNSUPPORTED;
    if (num_seqs == 0) return FNPU_OK;
    if (max_context_len < 1 || split_keys < 0 || (split_keys % 64) != 0) return FNPU_EINVAL;
    if (split_keys == 0) split_keys = 512;
    if (block_table_stride < (max_context_len + desc->block_size - 1) / desc->block_size)
        return FNPU_EINVAL;
    if (!context_len || !block_table || !q || !k_cache || !v_cache || !out || !lse) return FNPU_EINVAL;
    const uintptr_t mis = reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k_cache) |
                          reinterpret_cast<uintptr_t>(v_cache) | reinterpret_cast<uintptr_t>(out) |
                          reinterpret_cast<uintptr_t>(lse);
    if (mis & 15u) return FNPU_EINVAL;

    const int32_t G = Hq / Hkv;
    const int64_t max_splits = (max_context_len + split_keys - 1) / split_keys;
    const int64_t groups = static_cast<int64_t>(num_seqs) * Hkv;
    const int64_t parts = groups * max_splits;
    // scratch layout (floats): counters | part_lse | part_o, each 64-float aligned
    const int64_t n_cnt = (groups + 63) / 64 * 64;
    const int64_t n_lse = (parts * G + 63) / 64 * 64;
    const int64_t n_o = parts * G * D;
    if (n_cnt + n_lse + n_o > static_cast<int64_t>(kScratchFloats) || groups * max_splits > INT32_MAX)
        return FNPU_EINVAL;  // needs more than FNPU_NOALLOC_SCRATCH_BYTES

    float *scratch = nullptr;
    int rc = scratch_address(&scratch);
    if (rc != FNPU_OK) return rc;
    int *err = nullptr;
    rc = global_error_address(&err);
    if (rc != FNPU_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(scratch, 0, sizeof(int32_t) * static_cast<size_t>(groups), st) != cudaSuccess)
        return FNPU_ECUDA;

    NoallocParams p = {};
    p.q = static_cast<const __nv_bfloat16 *>(q);
    p.k_cache = static_cast<const __nv_bfloat16 *>(k_cache);
    p.v_cache = static_cast<const __nv_bfloat16 *>(v_cache);
    p.out = static_cast<__nv_bfloat16 *>(out);
    p.lse = lse;
    p.context_len = context_len;
    p.block_table = block_table;
    p.bt_stride = block_table_stride;
    p.num_q_heads = Hq;
    p.num_kv_heads = Hkv;
    p.group = G;
    p.block_size = desc->block_size;
    p.max_splits = static_cast<int32_t>(max_splits);
    p.split_keys = split_keys;
    p.max_context_len = max_context_len;
    p.num_blocks = desc->num_blocks;
    p.err = err;
    p.k_slot_stride = static_cast<int64_t>(Hkv) * D;
    p.v_slot_stride = static_cast<int64_t>(Hkv) * D;
    const float scale = desc->softmax_scale > 0.f ? desc->softmax_scale
                                                  : static_cast<float>(1.0 / sqrt(static_cast<double>(D)));
    p.scale_log2 = scale * 1.4426950408889634f;
    p.counters = reinterpret_cast<int32_t *>(scratch);
    p.part_lse = scratch + n_cnt;
    p.part_o = scratch + n_cnt + n_lse;
    const int grid = static_cast<int>(parts);
    return D == 64 ? launch_noalloc<64>(p, grid, st) : launch_noalloc<128>(p, grid, st);
}
