// qx_attn.cu -- the single-head attention core O = (Q K^T) V, no softmax and
// no scale (paper: Methodology; Table 2 attention rows), as two chained
// products on the tiled substrate with S = Q K^T kept on chip.
//
// Grid: query tiles (128 queries) x key splits; the splits of one query tile
// form one thread-block cluster.  Each CTA walks its run of key blocks:
//   1. S_b = Q K_b^T        tcgen05 into TMEM (M = 128 queries, N = keys);
//   2. S_b -> operand       each thread reads its query row of S from TMEM and
//                           writes it back to shared memory as the operand of
//                           the second product (K-major, 128B-swizzled);
//   3. O^T += V_b^T S_b^T   tcgen05 into TMEM (M = 128 rows of V^T, i.e. the d
//                           outputs padded with zeros; N = 2 x 128 queries).
// At the end every CTA leaves its partial O in its own shared memory; after a
// cluster barrier, CTA r of the cluster adds slice r of the query rows over
// all CTAs of the cluster (distributed shared memory, fixed rank order) and
// writes O.  No atomics, no zeroing, and the same order on every run.
//
// Integer kind (FP16 digits, exact): S is exact because the plan bounds
// d * max|Q| * max|K| by 2^24; S is split into two balanced digits (rows
// 0-127 low, 128-255 high of the N-side tile) and the plan bounds
// keys-per-CTA * max|digit| * max|V| by 2^24, so O^T's FP32 sums are exact;
// O = lo + (hi << shift) in wrapping int32.
//
// FP32 kind (3xTF32, kind::tf32): every operand is split into TF32 big +
// small parts; S_b = Q_big [K_big; K_small]^T + Q_small K_big^T and
// O^T += V_big^T [S_big; S_small]^T + V_small^T S_big^T, with S split on
// chip.  Key blocks hold 32 keys (one 128-byte FP32 row).
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "qx_device.cuh"
#include "qx_internal.h"

namespace qx {

namespace attn {
constexpr int kThreads = 160;       // warps 0-3: S conversion and epilogue; warp 4: TMA + MMA
constexpr int kConv = 128;          // one converter thread per query row
constexpr int kQTile = 128;         // queries per CTA
constexpr int kTmemCols = 512;
constexpr int kTmemS = 0;           // S block
constexpr int kTmemO = 256;         // O^T: 256 columns (two halves of 128 queries)
constexpr int kMaxCluster = 8;

// Integer kind
constexpr int kKeys = 64;
constexpr uint32_t kIdescS = make_idesc(128, kKeys, 0);
constexpr uint32_t kIdescO = make_idesc(128, 256, 0);
struct Smem {
    static constexpr int Q_BLK = kQTile * 128;          // one 64-wide k-block of Q
    static constexpr int K_BLK = kKeys * 128;           // one 64-wide k-block of K
    static constexpr int VT = 128 * 128;                // 128 rows of V^T x 64 keys
    static constexpr int S = 256 * 128;                 // both digit tiles
    static constexpr int KV_STAGE = 2 * K_BLK + VT;     // K (up to 2 k-blocks) + V^T
    static constexpr int q_off = 0;                     // Q: up to 2 k-blocks
    static constexpr int kv_off = 2 * Q_BLK;
    static constexpr int s_off = kv_off + 2 * KV_STAGE;
    static constexpr int part_off = s_off + S;          // partial O: 128 x (64 or 128) int32
    static constexpr int bar_off = part_off + kQTile * 128 * 4;
    static constexpr int total = bar_off + 256 + 1024;
};

// FP32 kind
constexpr int kKeys32 = 32;
constexpr int kDp32 = 64;                               // head size padded to 64
constexpr uint32_t kIdescS32 = make_idesc(128, 2 * kKeys32, 2);
constexpr uint32_t kIdescS32First = make_idesc(128, kKeys32, 2);
constexpr uint32_t kIdescO32 = make_idesc(128, 256, 2);
constexpr uint32_t kIdescO32First = make_idesc(128, 128, 2);
struct Smem32 {
    static constexpr int Q_KQ = 2 * kQTile * 128;       // one 32-wide k-block, big + small
    static constexpr int K_KQ = 2 * kKeys32 * 128;      // one 32-wide k-block, big + small
    static constexpr int VT = 2 * 128 * 128;            // big + small, 128 rows, 32 keys
    static constexpr int KV_STAGE = 2 * K_KQ + VT;
    static constexpr int S = 2 * kQTile * 128;
    static constexpr int q_off = 0;
    static constexpr int kv_off = 2 * Q_KQ;
    static constexpr int s_off = kv_off + 2 * KV_STAGE;
    static constexpr int part_off = s_off;              // partial O reuses the S tile at the end
    static constexpr int bar_off = s_off + S;
    static constexpr int total = bar_off + 256 + 1024;
};
static_assert(kQTile * kDp32 * 4 <= Smem32::S, "FP32 partial must fit the S tile");

struct Bars {
    uint64_t *q, *kv, *s, *sready, *o, *tail;
    uint32_t *tmem_slot;
    volatile int *abort_flag;
    __device__ Bars(uint8_t *base) {
        uint64_t *b = reinterpret_cast<uint64_t *>(base);
        q = b;
        kv = b + 1;   // [2]
        s = b + 3;
        sready = b + 4;
        o = b + 5;
        tail = b + 6;
        tmem_slot = reinterpret_cast<uint32_t *>(b + 8);
        abort_flag = reinterpret_cast<volatile int *>(b + 9);
    }
    __device__ void init() {
        mbar_init(q, 1);
        mbar_init(&kv[0], 1);
        mbar_init(&kv[1], 1);
        mbar_init(s, 1);
        mbar_init(sready, kConv);
        mbar_init(o, 1);
        mbar_init(tail, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
};

// After an abort: let issued MMAs and copies land before resources go away.
__device__ __forceinline__ void drain_after_abort(const Bars &b, int issued_kv) {
    tc_commit(b.tail);
    mbar_wait_drain(b.tail, 0);
    for (int s = 0; s < 2; ++s) {
        const int uses = issued_kv / 2 + (s < issued_kv % 2 ? 1 : 0);
        if (uses > 0) mbar_wait_drain(&b.kv[s], uint32_t((uses - 1) & 1));
    }
    mbar_wait_drain(b.q, 0);
}

// Cluster reduction: CTA `rank` adds its slice of the 128 query rows over all
// `cs` CTAs (rank order) and writes O rows qt*128 + j.  part is [128][pd].
template <bool FLOAT>
__device__ __forceinline__ void cluster_reduce_store(const void *part, int pd, int cs, int qt,
                                                     const AttnArgs &a) {
    const uint32_t rank = cluster_rank();
    const int rows = (kQTile + cs - 1) / cs;
    const int j0 = int(rank) * rows;
    const int j1 = min(kQTile, j0 + rows);
    const uint32_t pbase = smem_addr(part);
    for (int idx = threadIdx.x; idx < (j1 - j0) * a.d; idx += blockDim.x) {
        const int j = j0 + idx / a.d;
        const int c = idx - (idx / a.d) * a.d;
        const int q = qt * kQTile + j;
        if (q >= a.L) continue;
        const uint32_t off = uint32_t(j * pd + c) * 4u;
        if constexpr (FLOAT) {
            float acc = 0.f;
            for (int src = 0; src < cs; ++src)
                acc += __uint_as_float(ld_cluster_u32(cluster_map(pbase + off, uint32_t(src))));
            static_cast<float *>(a.out)[int64_t(q) * a.d + c] = acc;
        } else {
            uint32_t acc = 0u;
            for (int src = 0; src < cs; ++src) acc += ld_cluster_u32(cluster_map(pbase + off, uint32_t(src)));
            static_cast<int32_t *>(a.out)[int64_t(q) * a.d + c] = int32_t(acc);
        }
    }
}
}  // namespace attn

// ==================================================================== integer
__global__ void __launch_bounds__(attn::kThreads, 1) attn_core_kernel(const __grid_constant__ AttnArgs a) {
    using namespace attn;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sq = smem + Smem::q_off;
    uint8_t *skv = smem + Smem::kv_off;
    uint8_t *ss = smem + Smem::s_off;
    int32_t *part = reinterpret_cast<int32_t *>(smem + Smem::part_off);
    Bars bar(smem + Smem::bar_off);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int cs = a.key_splits;                         // cluster size
    const int qt = blockIdx.x / cs;
    const int split = blockIdx.x - qt * cs;
    const int dkb = a.d > 64 ? 2 : 1;                    // 64-wide k-blocks of Q and K
    const int pd = a.d > 64 ? 128 : 64;                  // row pitch of the partial O
    const int key_begin = split * a.keys_per_split;
    int nkb = (min(a.L, key_begin + a.keys_per_split) - key_begin + kKeys - 1) / kKeys;
    if (nkb < 0) nkb = 0;

    if (threadIdx.x == 0) bar.init();
    if (warp == 4) {
        tmem_alloc(bar.tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *bar.tmem_slot;
    const uint32_t tS = tmem + kTmemS;
    const uint32_t tO = tmem + kTmemO;
    pdl_wait();   // packed operands come from the kernel launched just before

    bool ok = true;
    if (warp == 4) {
        if (lane == 0 && nkb > 0) {
            // ------------------------------------------- loads + MMA issue
            tma_prefetch(&a.tm_q);
            tma_prefetch(&a.tm_k);
            tma_prefetch(&a.tm_vt);
            mbar_expect_tx(bar.q, dkb * Smem::Q_BLK);
            for (int kb = 0; kb < dkb; ++kb)
                tma_load_2d(sq + kb * Smem::Q_BLK, &a.tm_q, bar.q, kb * 64, qt * kQTile);
            auto load_kv = [&](int b) {
                uint8_t *st = skv + (b & 1) * Smem::KV_STAGE;
                const int key0 = key_begin + b * kKeys;
                mbar_expect_tx(&bar.kv[b & 1], dkb * Smem::K_BLK + Smem::VT);
                for (int kb = 0; kb < dkb; ++kb)
                    tma_load_2d(st + kb * Smem::K_BLK, &a.tm_k, &bar.kv[b & 1], kb * 64, key0);
                tma_load_2d(st + 2 * Smem::K_BLK, &a.tm_vt, &bar.kv[b & 1], key0, 0);
            };
            load_kv(0);
            int issued_kv = 1;
            for (int b = 0; ok && b < nkb; ++b) {
                if (b + 1 < nkb) {
                    // stage (b+1)&1 was read by block b-1; its O MMA must be done
                    if (b >= 1 && !mbar_wait(bar.o, uint32_t((b - 1) & 1), bar.abort_flag, a.err)) {
                        ok = false;
                        break;
                    }
                    load_kv(b + 1);
                    ++issued_kv;
                }
                if (b == 0 && !mbar_wait(bar.q, 0, bar.abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                if (!mbar_wait(&bar.kv[b & 1], uint32_t((b >> 1) & 1), bar.abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t qa = smem_addr(sq);
                const uint32_t ka = smem_addr(skv + (b & 1) * Smem::KV_STAGE);
                for (int kb = 0; kb < dkb; ++kb)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        mma_f16(tS, make_sdesc(qa + kb * Smem::Q_BLK + kk * 32),
                                make_sdesc(ka + kb * Smem::K_BLK + kk * 32), kIdescS,
                                (kb > 0 || kk > 0) ? 1u : 0u);
                tc_commit(bar.s);
                if (!mbar_wait(bar.sready, uint32_t(b & 1), bar.abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t va = ka + 2 * Smem::K_BLK;
                const uint32_t sa = smem_addr(ss);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    mma_f16(tO, make_sdesc(va + kk * 32), make_sdesc(sa + kk * 32), kIdescO,
                            (b > 0 || kk > 0) ? 1u : 0u);
                tc_commit(bar.o);
            }
            if (!ok) drain_after_abort(bar, issued_kv);
        }
    } else {
        // ------------------------------------------- S -> FP16 digits in smem
        const int row = warp * 32 + lane;                // query row of this thread
        const int half = 1 << (a.s_shift - 1);
        const int mask = (1 << a.s_shift) - 1;
        for (int b = 0; b < nkb; ++b) {
            if (!mbar_wait(bar.s, uint32_t(b & 1), bar.abort_flag, a.err)) {
                ok = false;
                break;
            }
            if (b >= 1 && !mbar_wait(bar.o, uint32_t((b - 1) & 1), bar.abort_flag, a.err)) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint8_t *rlo = ss + row * 128;
            uint8_t *rhi = ss + (128 + row) * 128;
#pragma unroll
            for (int p = 0; p < kKeys / 32; ++p) {
                uint32_t v[32];
                tmem_ld32(tS + (uint32_t(warp * 32) << 16) + p * 32, v);
                tmem_wait_ld(v);
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    __align__(16) __half lo[8], hi[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int32_t sv = __float2int_rn(__uint_as_float(v[c * 8 + e]));
                        const int32_t d0 = ((sv + half) & mask) - half;
                        lo[e] = __int2half_rn(d0);
                        hi[e] = __int2half_rn((sv - d0) >> a.s_shift);
                    }
                    const int chunk = p * 4 + c;                     // 16-byte chunk of the row
                    const int pos = (chunk ^ (row & 7)) << 4;        // 128B swizzle
                    *reinterpret_cast<uint4 *>(rlo + pos) = *reinterpret_cast<uint4 *>(lo);
                    *reinterpret_cast<uint4 *>(rhi + pos) = *reinterpret_cast<uint4 *>(hi);
                }
            }
            // generic-proxy smem writes -> visible to the tensor core's async proxy
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            tc_fence_before();
            mbar_arrive(bar.sready);
        }
        // ------------------------------- this CTA's partial O -> shared memory
        const int c = warp * 32 + lane;                  // output column (row of V^T)
        const bool have = ok && nkb > 0 && mbar_wait(bar.o, uint32_t((nkb - 1) & 1), bar.abort_flag, a.err);
        if (have) tc_fence_after();
        if (warp * 32 < a.d) {
#pragma unroll 1
            for (int p = 0; p < kQTile / 32; ++p) {
                uint32_t lo[32], hi[32];
                if (have) {
                    tmem_ld32(tO + (uint32_t(warp * 32) << 16) + p * 32, lo);
                    tmem_wait_ld(lo);
                    tmem_ld32(tO + (uint32_t(warp * 32) << 16) + 128 + p * 32, hi);
                    tmem_wait_ld(hi);
                }
#pragma unroll
                for (int x = 0; x < 32; ++x) {
                    const uint32_t val =
                        have ? uint32_t(__float2int_rn(__uint_as_float(lo[x]))) +
                                   (uint32_t(__float2int_rn(__uint_as_float(hi[x]))) << a.s_shift)
                             : 0u;
                    if (c < a.d) part[(p * 32 + x) * pd + c] = int32_t(val);
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync();                                      // every partial is in place
    cluster_reduce_store<false>(part, pd, cs, qt, a);
    cluster_sync();                                      // peers are done reading
    if (warp == 4) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ======================================================================= FP32
__global__ void __launch_bounds__(attn::kThreads, 1)
    attn_core_f32_kernel(const __grid_constant__ AttnArgs a) {
    using namespace attn;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sq = smem + Smem32::q_off;
    uint8_t *skv = smem + Smem32::kv_off;
    uint8_t *ss = smem + Smem32::s_off;
    float *part = reinterpret_cast<float *>(smem + Smem32::part_off);
    Bars bar(smem + Smem32::bar_off);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int cs = a.key_splits;
    const int qt = blockIdx.x / cs;
    const int split = blockIdx.x - qt * cs;
    const int key_begin = split * a.keys_per_split;
    int nkb = (min(a.L, key_begin + a.keys_per_split) - key_begin + kKeys32 - 1) / kKeys32;
    if (nkb < 0) nkb = 0;

    if (threadIdx.x == 0) bar.init();
    if (warp == 4) {
        tmem_alloc(bar.tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *bar.tmem_slot;
    const uint32_t tS = tmem + kTmemS;
    const uint32_t tO = tmem + kTmemO;
    pdl_wait();   // packed operands come from the kernel launched just before

    bool ok = true;
    if (warp == 4) {
        if (lane == 0 && nkb > 0) {
            tma_prefetch(&a.tm_q);
            tma_prefetch(&a.tm_k);
            tma_prefetch(&a.tm_vt);
            mbar_expect_tx(bar.q, 2 * Smem32::Q_KQ);
            for (int kq = 0; kq < 2; ++kq)
                tma_load_3d(sq + kq * Smem32::Q_KQ, &a.tm_q, bar.q, kq * 32, qt * kQTile, 0);
            auto load_kv = [&](int b) {
                uint8_t *st = skv + (b & 1) * Smem32::KV_STAGE;
                const int key0 = key_begin + b * kKeys32;
                mbar_expect_tx(&bar.kv[b & 1], Smem32::KV_STAGE);
                for (int kq = 0; kq < 2; ++kq)
                    tma_load_3d(st + kq * Smem32::K_KQ, &a.tm_k, &bar.kv[b & 1], kq * 32, key0, 0);
                tma_load_3d(st + 2 * Smem32::K_KQ, &a.tm_vt, &bar.kv[b & 1], key0, 0, 0);
            };
            load_kv(0);
            int issued_kv = 1;
            for (int b = 0; ok && b < nkb; ++b) {
                if (b + 1 < nkb) {
                    if (b >= 1 && !mbar_wait(bar.o, uint32_t((b - 1) & 1), bar.abort_flag, a.err)) {
                        ok = false;
                        break;
                    }
                    load_kv(b + 1);
                    ++issued_kv;
                }
                if (b == 0 && !mbar_wait(bar.q, 0, bar.abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                if (!mbar_wait(&bar.kv[b & 1], uint32_t((b >> 1) & 1), bar.abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t qa = smem_addr(sq);
                const uint32_t ka = smem_addr(skv + (b & 1) * Smem32::KV_STAGE);
                for (int kq = 0; kq < 2; ++kq)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint32_t qb = qa + kq * Smem32::Q_KQ + kk * 32;
                        const uint64_t kd = make_sdesc(ka + kq * Smem32::K_KQ + kk * 32);
                        mma_tf32(tS, make_sdesc(qb), kd, kIdescS32, (kq > 0 || kk > 0) ? 1u : 0u);
                        mma_tf32(tS, make_sdesc(qb + kQTile * 128), kd, kIdescS32First, 1u);
                    }
                tc_commit(bar.s);
                if (!mbar_wait(bar.sready, uint32_t(b & 1), bar.abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t va = ka + 2 * Smem32::K_KQ;
                const uint32_t sa = smem_addr(ss);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const uint64_t sd = make_sdesc(sa + kk * 32);
                    mma_tf32(tO, make_sdesc(va + kk * 32), sd, kIdescO32, (b > 0 || kk > 0) ? 1u : 0u);
                    mma_tf32(tO, make_sdesc(va + 128 * 128 + kk * 32), sd, kIdescO32First, 1u);
                }
                tc_commit(bar.o);
            }
            if (!ok) drain_after_abort(bar, issued_kv);
        }
    } else {
        // ---------------------------------------- S -> TF32 big/small in smem
        const int row = warp * 32 + lane;
        for (int b = 0; b < nkb; ++b) {
            if (!mbar_wait(bar.s, uint32_t(b & 1), bar.abort_flag, a.err)) {
                ok = false;
                break;
            }
            if (b >= 1 && !mbar_wait(bar.o, uint32_t((b - 1) & 1), bar.abort_flag, a.err)) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint32_t v0[32], v1[32];
            tmem_ld32(tS + (uint32_t(warp * 32) << 16), v0);
            tmem_ld32(tS + (uint32_t(warp * 32) << 16) + kKeys32, v1);
            tmem_wait_ld(v0);
            tmem_wait_ld(v1);
            uint8_t *rbig = ss + row * 128;
            uint8_t *rsmall = ss + (kQTile + row) * 128;
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                __align__(16) float big[4], small[4];
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    tf32_split(__uint_as_float(v0[c * 4 + e]) + __uint_as_float(v1[c * 4 + e]),
                               big[e], small[e]);
                const int pos = (c ^ (row & 7)) << 4;
                *reinterpret_cast<uint4 *>(rbig + pos) = *reinterpret_cast<uint4 *>(big);
                *reinterpret_cast<uint4 *>(rsmall + pos) = *reinterpret_cast<uint4 *>(small);
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            tc_fence_before();
            mbar_arrive(bar.sready);
        }
        // ------------------------------- this CTA's partial O -> shared memory
        // (the S tile is free once the last O MMA has completed)
        const int c = warp * 32 + lane;
        const bool have = ok && nkb > 0 && mbar_wait(bar.o, uint32_t((nkb - 1) & 1), bar.abort_flag, a.err);
        if (have) tc_fence_after();
        if (warp * 32 < kDp32) {
#pragma unroll 1
            for (int p = 0; p < kQTile / 32; ++p) {
                uint32_t lo[32], hi[32];
                if (have) {
                    tmem_ld32(tO + (uint32_t(warp * 32) << 16) + p * 32, lo);
                    tmem_ld32(tO + (uint32_t(warp * 32) << 16) + 128 + p * 32, hi);
                    tmem_wait_ld(lo);
                    tmem_wait_ld(hi);
                }
#pragma unroll
                for (int x = 0; x < 32; ++x)
                    part[(p * 32 + x) * kDp32 + c] =
                        have ? __uint_as_float(lo[x]) + __uint_as_float(hi[x]) : 0.f;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync();
    cluster_reduce_store<true>(part, kDp32, cs, qt, a);
    cluster_sync();
    if (warp == 4) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ------------------------------------------------------------------- host
cudaError_t attn_prepare() {
    return cudaFuncSetAttribute(attn_core_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                attn::Smem::total);
}

cudaError_t attn_launch(const AttnArgs &a, cudaStream_t stream) {
    return launch_pdl(attn_core_kernel, a.q_tiles * a.key_splits, attn::kThreads, attn::Smem::total,
                      stream, a, a.key_splits);
}

cudaError_t attn_f32_prepare() {
    return cudaFuncSetAttribute(attn_core_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                attn::Smem32::total);
}

cudaError_t attn_f32_launch(const AttnArgs &a, cudaStream_t stream) {
    return launch_pdl(attn_core_f32_kernel, a.q_tiles * a.key_splits, attn::kThreads,
                      attn::Smem32::total, stream, a, a.key_splits);
}

int attn_max_cluster() { return attn::kMaxCluster; }

}  // namespace qx
