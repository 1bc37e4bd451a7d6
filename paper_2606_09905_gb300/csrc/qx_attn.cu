// qx_attn.cu -- the single-head attention core O = (Q K^T) V, no softmax and
// no scale (paper: Methodology; Table 2 attention rows), as two chained
// products on the tiled substrate with S = Q K^T kept on chip.
//
// One CTA owns a tile of 128 queries and a run of key blocks (64 keys each):
//   1. S_b = Q K_b^T        tcgen05 kind::f16 (M = 128 queries, N = 64 keys),
//                           FP32 accumulator in TMEM; exact because the plan
//                           bounds d * max|Q| * max|K| by 2^24.
//   2. S_b -> limbs         each thread reads its query row of S from TMEM,
//                           converts it to int32 (exact), splits it into two
//                           balanced digits and writes them as FP16 into a
//                           K-major, 128-byte-swizzled shared-memory tile
//                           (rows 0-127 low digit, rows 128-255 high digit).
//   3. O^T += V_b^T S_b^T   tcgen05 kind::f16 (M = 128 rows of V^T, i.e. the
//                           d outputs padded to 128 with zeros; N = 256 =
//                           both digits of the 128 queries; K = 64 keys).
//                           The plan bounds keys-per-CTA * max|digit| * max|V|
//                           by 2^24, so the FP32 sums stay exact.
//   4. epilogue             O = lo + (hi << shift) in int32; each thread owns
//                           one output column c, so a warp's atomic adds cover
//                           32 consecutive int32 values of one query row.
// CTAs that share a query tile but own different key runs add their partial
// O with integer atomics: exact, so the result does not depend on order.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "qx_device.cuh"
#include "qx_internal.h"

namespace qx {

namespace attn {
constexpr int kThreads = 160;                   // warps 0-3 convert/store, warp 4 issues
constexpr int kConv = 128;                      // converter threads (one per query row)
constexpr int kKeys = 64;                       // keys per block
constexpr int kQTile = 128;                     // queries per CTA
constexpr int kTmemCols = 512;
constexpr int kTmemS = 0;                       // S block: 64 columns
constexpr int kTmemO = 256;                     // O^T: 256 columns (lo | hi)
constexpr uint32_t kIdescS = make_idesc(128, kKeys, 0);
constexpr uint32_t kIdescO = make_idesc(128, 256, 0);

struct Smem {
    // every operand tile starts on a 1024-byte boundary (128B swizzle atoms)
    static constexpr int Q_BLK = kQTile * 128;          // one 64-wide k-block of Q
    static constexpr int K_BLK = kKeys * 128;           // one 64-wide k-block of K
    static constexpr int VT = 128 * 128;                // 128 rows of V^T x 64 keys
    static constexpr int S = 256 * 128;                 // both digit tiles
    static constexpr int q_off = 0;                      // Q: up to 2 k-blocks
    static constexpr int kv_off = 2 * Q_BLK;
    static constexpr int KV_STAGE = 2 * K_BLK + VT;      // K (up to 2 k-blocks) + V^T
    static constexpr int s_off = 2 * Q_BLK + 2 * KV_STAGE;
    static constexpr int bar_off = s_off + S;
    static constexpr int total = bar_off + 256 + 1024;
};
}  // namespace attn

__global__ void __launch_bounds__(attn::kThreads, 1) attn_core_kernel(const __grid_constant__ AttnArgs a) {
    using namespace attn;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sq = smem + Smem::q_off;
    uint8_t *skv = smem + Smem::kv_off;
    uint8_t *ss = smem + Smem::s_off;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + Smem::bar_off);
    uint64_t *bar_q = bars + 0;
    uint64_t *bar_kv = bars + 1;      // [2]
    uint64_t *bar_s = bars + 3;
    uint64_t *bar_sready = bars + 4;
    uint64_t *bar_o = bars + 5;
    uint64_t *bar_tail = bars + 6;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 8);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bars + 9);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int qt = blockIdx.x % a.q_tiles;
    const int split = blockIdx.x / a.q_tiles;
    const int dkb = a.d > 64 ? 2 : 1;                    // 64-wide k-blocks of Q and K
    const int key_begin = split * a.keys_per_split;
    int nkb = (min(a.L, key_begin + a.keys_per_split) - key_begin + kKeys - 1) / kKeys;
    if (nkb < 0) nkb = 0;

    if (threadIdx.x == 0) {
        mbar_init(bar_q, 1);
        mbar_init(&bar_kv[0], 1);
        mbar_init(&bar_kv[1], 1);
        mbar_init(bar_s, 1);
        mbar_init(bar_sready, kConv);
        mbar_init(bar_o, 1);
        mbar_init(bar_tail, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 4) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t tS = tmem + kTmemS;
    const uint32_t tO = tmem + kTmemO;

    bool ok = true;
    if (warp == 4) {
      if (lane == 0 && nkb > 0) {
        // ------------------------------------------- loads + MMA issue
        tma_prefetch(&a.tm_q);
        tma_prefetch(&a.tm_k);
        tma_prefetch(&a.tm_vt);
        mbar_expect_tx(bar_q, dkb * Smem::Q_BLK);
        for (int kb = 0; kb < dkb; ++kb)
            tma_load_2d(sq + kb * Smem::Q_BLK, &a.tm_q, bar_q, kb * 64, qt * kQTile);
        auto load_kv = [&](int b) {
            uint8_t *st = skv + (b & 1) * Smem::KV_STAGE;
            const int key0 = key_begin + b * kKeys;
            mbar_expect_tx(&bar_kv[b & 1], dkb * Smem::K_BLK + Smem::VT);
            for (int kb = 0; kb < dkb; ++kb)
                tma_load_2d(st + kb * Smem::K_BLK, &a.tm_k, &bar_kv[b & 1], kb * 64, key0);
            tma_load_2d(st + 2 * Smem::K_BLK, &a.tm_vt, &bar_kv[b & 1], key0, 0);
        };
        load_kv(0);
        int issued_kv = 1;
        for (int b = 0; ok && b < nkb; ++b) {
            if (b + 1 < nkb) {
                // stage (b+1)&1 was read by block b-1; its O MMA must be done
                if (b >= 1 && !mbar_wait(bar_o, uint32_t((b - 1) & 1), abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                load_kv(b + 1);
                ++issued_kv;
            }
            if (b == 0 && !mbar_wait(bar_q, 0, abort_flag, a.err)) {
                ok = false;
                break;
            }
            if (!mbar_wait(&bar_kv[b & 1], uint32_t((b >> 1) & 1), abort_flag, a.err)) {
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
            tc_commit(bar_s);
            if (!mbar_wait(bar_sready, uint32_t(b & 1), abort_flag, a.err)) {
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
            tc_commit(bar_o);
        }
        if (!ok) {
            tc_commit(bar_tail);
            mbar_wait_drain(bar_tail, 0);
            for (int s = 0; s < 2; ++s) {
                const int uses = issued_kv / 2 + (s < issued_kv % 2 ? 1 : 0);
                if (uses > 0) mbar_wait_drain(&bar_kv[s], uint32_t((uses - 1) & 1));
            }
            mbar_wait_drain(bar_q, 0);
        }
      }
    } else {
    // ------------------------------------------- S -> FP16 digits in smem
    const int row = warp * 32 + lane;                    // query row of this thread
    const int half = 1 << (a.s_shift - 1);
    const int mask = (1 << a.s_shift) - 1;
    for (int b = 0; b < nkb; ++b) {
        if (!mbar_wait(bar_s, uint32_t(b & 1), abort_flag, a.err)) {
            ok = false;
            break;
        }
        if (b >= 1 && !mbar_wait(bar_o, uint32_t((b - 1) & 1), abort_flag, a.err)) {
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
        mbar_arrive(bar_sready);
    }

    // ------------------------------------------- epilogue: O += lo + hi<<s
    if (ok && nkb > 0 && mbar_wait(bar_o, uint32_t((nkb - 1) & 1), abort_flag, a.err)) {
        tc_fence_after();
        const int c = warp * 32 + lane;                  // output column (row of V^T)
        if (warp * 32 < a.d) {
#pragma unroll 1
            for (int p = 0; p < kQTile / 32; ++p) {
                uint32_t lo[32], hi[32];
                tmem_ld32(tO + (uint32_t(warp * 32) << 16) + p * 32, lo);
                tmem_wait_ld(lo);
                tmem_ld32(tO + (uint32_t(warp * 32) << 16) + 128 + p * 32, hi);
                tmem_wait_ld(hi);
#pragma unroll
                for (int x = 0; x < 32; ++x) {
                    const int qrow = qt * kQTile + p * 32 + x;
                    const uint32_t val = uint32_t(__float2int_rn(__uint_as_float(lo[x]))) +
                                         (uint32_t(__float2int_rn(__uint_as_float(hi[x])))
                                          << a.s_shift);
                    if (c < a.d && qrow < a.L)
                        atomicAdd(static_cast<int32_t *>(a.out) + int64_t(qrow) * a.d + c, int32_t(val));
                }
            }
        }
    }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 4) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ===================================================================== FP32
// The FP32 attention core (Table 2, attention FP32 row) on the same two-MMA
// structure with kind::tf32 and a 3xTF32 split of every operand:
//   S_b = Q_big [K_big; K_small]^T + Q_small K_big^T          (two MMAs)
//   O^T += V_big^T [S_big; S_small]^T + V_small^T S_big^T     (two MMAs)
// where S is split into TF32 big + small parts on chip.  Key blocks hold 32
// keys (one 128-byte FP32 row).  Each CTA writes its partial O to the
// workspace; the last CTA of a query tile to finish (arrival counter) adds
// the partials in split order, so the result does not depend on timing.
namespace attn32 {
constexpr int kThreads = 160;
constexpr int kConv = 128;
constexpr int kKeys = 32;
constexpr int kQTile = 128;
constexpr int kDp = 64;                         // head size padded to 64
constexpr int kTmemCols = 512;
constexpr int kTmemS = 0;                       // [Qb.Kb | Qb.Ks], + Qs.Kb on the first 32
constexpr int kTmemO = 256;                     // [Vb.Sb | Vb.Ss], + Vs.Sb on the first 128
constexpr uint32_t kIdescS = make_idesc(128, 2 * kKeys, 2);
constexpr uint32_t kIdescS1 = make_idesc(128, kKeys, 2);
constexpr uint32_t kIdescO = make_idesc(128, 256, 2);
constexpr uint32_t kIdescO1 = make_idesc(128, 128, 2);

struct Smem {
    static constexpr int Q_KQ = 2 * kQTile * 128;        // one 32-wide k-block, both limbs
    static constexpr int K_KQ = 2 * kKeys * 128;         // one 32-wide k-block, both limbs
    static constexpr int VT = 2 * 128 * 128;             // both limbs, 128 rows, 32 keys
    static constexpr int KV_STAGE = 2 * K_KQ + VT;
    static constexpr int S = 2 * kQTile * 128;
    static constexpr int q_off = 0;
    static constexpr int kv_off = 2 * Q_KQ;
    static constexpr int s_off = kv_off + 2 * KV_STAGE;
    static constexpr int bar_off = s_off + S;
    static constexpr int total = bar_off + 256 + 1024;
};
}  // namespace attn32

__global__ void __launch_bounds__(attn32::kThreads, 1)
    attn_core_f32_kernel(const __grid_constant__ AttnArgs a) {
    using namespace attn32;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sq = smem + Smem::q_off;
    uint8_t *skv = smem + Smem::kv_off;
    uint8_t *ss = smem + Smem::s_off;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + Smem::bar_off);
    uint64_t *bar_q = bars + 0;
    uint64_t *bar_kv = bars + 1;      // [2]
    uint64_t *bar_s = bars + 3;
    uint64_t *bar_sready = bars + 4;
    uint64_t *bar_o = bars + 5;
    uint64_t *bar_tail = bars + 6;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 8);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(bars + 9);
    volatile int *is_last = reinterpret_cast<volatile int *>(bars + 10);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int qt = blockIdx.x % a.q_tiles;
    const int split = blockIdx.x / a.q_tiles;
    const int key_begin = split * a.keys_per_split;
    int nkb = (min(a.L, key_begin + a.keys_per_split) - key_begin + kKeys - 1) / kKeys;
    if (nkb < 0) nkb = 0;
    float *part = a.partial + (int64_t(qt) * a.key_splits + split) * kQTile * kDp;

    if (threadIdx.x == 0) {
        mbar_init(bar_q, 1);
        mbar_init(&bar_kv[0], 1);
        mbar_init(&bar_kv[1], 1);
        mbar_init(bar_s, 1);
        mbar_init(bar_sready, kConv);
        mbar_init(bar_o, 1);
        mbar_init(bar_tail, 1);
        *abort_flag = 0;
        *is_last = 0;
        fence_mbar_init();
    }
    if (warp == 4) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t tS = tmem + kTmemS;
    const uint32_t tO = tmem + kTmemO;

    bool ok = true;
    if (warp == 4) {
        if (lane == 0 && nkb > 0) {
            tma_prefetch(&a.tm_q);
            tma_prefetch(&a.tm_k);
            tma_prefetch(&a.tm_vt);
            mbar_expect_tx(bar_q, 2 * Smem::Q_KQ);
            for (int kq = 0; kq < 2; ++kq)
                tma_load_3d(sq + kq * Smem::Q_KQ, &a.tm_q, bar_q, kq * 32, qt * kQTile, 0);
            auto load_kv = [&](int b) {
                uint8_t *st = skv + (b & 1) * Smem::KV_STAGE;
                const int key0 = key_begin + b * kKeys;
                mbar_expect_tx(&bar_kv[b & 1], Smem::KV_STAGE);
                for (int kq = 0; kq < 2; ++kq)
                    tma_load_3d(st + kq * Smem::K_KQ, &a.tm_k, &bar_kv[b & 1], kq * 32, key0, 0);
                tma_load_3d(st + 2 * Smem::K_KQ, &a.tm_vt, &bar_kv[b & 1], key0, 0, 0);
            };
            load_kv(0);
            int issued_kv = 1;
            for (int b = 0; ok && b < nkb; ++b) {
                if (b + 1 < nkb) {
                    if (b >= 1 && !mbar_wait(bar_o, uint32_t((b - 1) & 1), abort_flag, a.err)) {
                        ok = false;
                        break;
                    }
                    load_kv(b + 1);
                    ++issued_kv;
                }
                if (b == 0 && !mbar_wait(bar_q, 0, abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                if (!mbar_wait(&bar_kv[b & 1], uint32_t((b >> 1) & 1), abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t qa = smem_addr(sq);
                const uint32_t ka = smem_addr(skv + (b & 1) * Smem::KV_STAGE);
                for (int kq = 0; kq < 2; ++kq)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint32_t qb = qa + kq * Smem::Q_KQ + kk * 32;
                        const uint64_t kd = make_sdesc(ka + kq * Smem::K_KQ + kk * 32);
                        mma_tf32(tS, make_sdesc(qb), kd, kIdescS, (kq > 0 || kk > 0) ? 1u : 0u);
                        mma_tf32(tS, make_sdesc(qb + kQTile * 128), kd, kIdescS1, 1u);
                    }
                tc_commit(bar_s);
                if (!mbar_wait(bar_sready, uint32_t(b & 1), abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t va = ka + 2 * Smem::K_KQ;
                const uint32_t sa = smem_addr(ss);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk) {
                    const uint64_t sd = make_sdesc(sa + kk * 32);
                    mma_tf32(tO, make_sdesc(va + kk * 32), sd, kIdescO, (b > 0 || kk > 0) ? 1u : 0u);
                    mma_tf32(tO, make_sdesc(va + 128 * 128 + kk * 32), sd, kIdescO1, 1u);
                }
                tc_commit(bar_o);
            }
            if (!ok) {
                tc_commit(bar_tail);
                mbar_wait_drain(bar_tail, 0);
                for (int s = 0; s < 2; ++s) {
                    const int uses = issued_kv / 2 + (s < issued_kv % 2 ? 1 : 0);
                    if (uses > 0) mbar_wait_drain(&bar_kv[s], uint32_t((uses - 1) & 1));
                }
                mbar_wait_drain(bar_q, 0);
            }
        }
    } else {
        // ---------------------------------------- S -> TF32 big/small in smem
        const int row = warp * 32 + lane;
        for (int b = 0; b < nkb; ++b) {
            if (!mbar_wait(bar_s, uint32_t(b & 1), abort_flag, a.err)) {
                ok = false;
                break;
            }
            if (b >= 1 && !mbar_wait(bar_o, uint32_t((b - 1) & 1), abort_flag, a.err)) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint32_t v0[32], v1[32];
            tmem_ld32(tS + (uint32_t(warp * 32) << 16), v0);
            tmem_ld32(tS + (uint32_t(warp * 32) << 16) + kKeys, v1);
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
            mbar_arrive(bar_sready);
        }
        // ---------------------------------------- partial O of this CTA
        const int c = warp * 32 + lane;
        if (ok && nkb > 0 && mbar_wait(bar_o, uint32_t((nkb - 1) & 1), abort_flag, a.err)) {
            tc_fence_after();
            if (warp * 32 < kDp) {
#pragma unroll 1
                for (int p = 0; p < kQTile / 32; ++p) {
                    uint32_t lo[32], hi[32];
                    tmem_ld32(tO + (uint32_t(warp * 32) << 16) + p * 32, lo);
                    tmem_ld32(tO + (uint32_t(warp * 32) << 16) + 128 + p * 32, hi);
                    tmem_wait_ld(lo);
                    tmem_wait_ld(hi);
#pragma unroll
                    for (int x = 0; x < 32; ++x)
                        part[(p * 32 + x) * kDp + c] = __uint_as_float(lo[x]) + __uint_as_float(hi[x]);
                }
            }
        } else if (nkb == 0 && warp * 32 < kDp) {
            for (int j = 0; j < kQTile; ++j) part[j * kDp + c] = 0.f;
        }
        __threadfence();
    }

    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && !*abort_flag) {
        const unsigned prev = atomicAdd(a.counters + qt, 1u);
        *is_last = prev == unsigned(a.key_splits - 1);
    }
    __syncthreads();
    if (*is_last) {
        // every split of this query tile has arrived: add them in split order
        __threadfence();
        float *out = static_cast<float *>(a.out);
        const float *base = a.partial + int64_t(qt) * a.key_splits * kQTile * kDp;
        for (int idx = threadIdx.x; idx < kQTile * a.d; idx += blockDim.x) {
            const int j = idx / a.d, c = idx - (idx / a.d) * a.d;
            const int q = qt * kQTile + j;
            if (q >= a.L) continue;
            float acc = 0.f;
            for (int sp = 0; sp < a.key_splits; ++sp)
                acc += __ldcg(base + (int64_t(sp) * kQTile + j) * kDp + c);
            out[int64_t(q) * a.d + c] = acc;
        }
    }
    if (warp == 4) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

cudaError_t attn_f32_prepare() {
    return cudaFuncSetAttribute(attn_core_f32_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                attn32::Smem::total);
}

cudaError_t attn_f32_launch(const AttnArgs &a, cudaStream_t stream) {
    attn_core_f32_kernel<<<a.q_tiles * a.key_splits, attn32::kThreads, attn32::Smem::total, stream>>>(a);
    return cudaGetLastError();
}

cudaError_t attn_prepare() {
    return cudaFuncSetAttribute(attn_core_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                attn::Smem::total);
}

cudaError_t attn_launch(const AttnArgs &a, cudaStream_t stream) {
    attn_core_kernel<<<a.q_tiles * a.key_splits, attn::kThreads, attn::Smem::total, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace qx
