// qx_attn_reassoc.cu -- the attention core in the reassociated order
// O = Q (K^T V), integer kinds only (Methodology: O = (Q K^T) V; matrix
// products associate exactly over the integers and modulo 2^32, so this is
// the same result with O(L d^2) instead of O(L^2 d) work, and S is never
// formed).
//
// One cluster of `cs` CTAs per head (grid x = cs, y = heads):
//   phase 1  CTA r sums W^T_r = V^T K over its run of keys on the tensor cores
//            (M = 128 rows of V^T, N = dp rows of K^T, 16 keys per MMA; both
//            packed transposed, keys contiguous).  The plan bounds the run so
//            max|K| max|V| keys < 2^24: the FP32 sums are exact integers.
//   reduce   rows of W^T are owned round the cluster: every CTA stores each
//            partial row into its owner's receive buffer (distributed shared
//            memory, fire-and-forget stores); the owner adds the cs copies
//            in rank order (wrapping int32), splits the rows into nd balanced
//            FP16 digits of `s_shift` bits and stores them into every CTA's
//            B operand of phase 2 (digits stacked along N).
//   phase 2  CTA r computes O rows of its query run, 128 at a time:
//            D = Q [W_0 | W_1 | ...] (M = 128 queries, N = nd dp, K = d), and
//            O = sum_t D_t << (t s) in wrapping int32.  The plan bounds
//            d max|Q| max|digit| by 2^24, so each D_t is exact.
// Warp 0 issues TMA loads, warp 1 owns TMEM and issues MMAs (as a converged
// warp, one elected lane), warps 2-9 (two per TMEM lane quarter, each taking
// half of the columns) drain the accumulators, reduce and write O.
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "qx_device.cuh"
#include "qx_internal.h"

namespace qx {

namespace ra {
constexpr int kThreads = 320;
constexpr int kProducerWarp = 0;
constexpr int kIssuerWarp = 1;
constexpr int kDrainWarps = 8;                          // warps 2-9
constexpr int kKeys = 64;
constexpr int kQTile = 128;
constexpr int kTmemCols = 512;
constexpr int kMaxStages = 6;
struct Smem {
    static constexpr int V_TILE = 128 * 128;            // phase 1 A: 128 rows of V^T x 64 keys
    static constexpr int RING = 128 * 1024;             // stages of V^T + K^T (phase 1) or Q (phase 2)
    static constexpr int ring_off = 0;
    static constexpr int dig_off = RING;                // W digits: dkb x (nd dp rows x 128 B)
    static constexpr int DIG = 64 * 1024;
    static constexpr int bar_off = dig_off + DIG;
    static constexpr int total = bar_off + 256 + 1024;
};
__host__ __device__ constexpr int wpitch(int dp) { return dp + 4; }   // int32 words per W^T row
// receive buffer: cs sources x ceil(dp / cs) rows x pitch, at most dp + cs - 1 rows
static_assert((128 + 7) * wpitch(128) * 4 <= Smem::RING, "receive buffer must fit the ring");
static_assert(Smem::total <= 227 * 1024, "shared memory");

struct Bars {
    uint64_t *full, *empty, *d1_full, *acc_full, *acc_empty, *tail;
    uint32_t *tmem_slot;
    volatile int *abort_flag;
    __device__ Bars(uint8_t *base) {
        uint64_t *b = reinterpret_cast<uint64_t *>(base);
        full = b;                              // [kMaxStages]
        empty = b + kMaxStages;                // [kMaxStages]
        d1_full = b + 2 * kMaxStages;
        acc_full = d1_full + 1;                // [2]
        acc_empty = acc_full + 2;              // [2]
        tail = acc_empty + 2;
        tmem_slot = reinterpret_cast<uint32_t *>(tail + 1);
        abort_flag = reinterpret_cast<volatile int *>(tail + 2);
    }
    __device__ void init() {
        for (int i = 0; i < kMaxStages; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        mbar_init(d1_full, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&acc_full[i], 1);
            mbar_init(&acc_empty[i], kDrainWarps);
        }
        mbar_init(tail, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
};
static_assert(2 * kMaxStages + 1 + 4 + 1 + 2 <= 256 / 8, "barrier block");
}  // namespace ra

__global__ void __launch_bounds__(ra::kThreads, 1) attn_reassoc_kernel(const __grid_constant__ AttnArgs a) {
    using namespace ra;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *ring = smem + Smem::ring_off;
    uint8_t *dig = smem + Smem::dig_off;
    int32_t *recv = reinterpret_cast<int32_t *>(ring);    // partial W^T rows this CTA owns, by source
    Bars bar(smem + Smem::bar_off);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int cs = a.key_splits;                        // cluster size = grid x
    const int rank = blockIdx.x;
    const int hd = blockIdx.y;
    const int dkb = a.d > 64 ? 2 : 1;
    const int dp = 64 * dkb;
    const int nd = a.ra_digits;
    const int pitch = wpitch(dp);
    const int stage_bytes = Smem::V_TILE + dp * 128;    // phase 2 uses dkb * 16 KB <= this
    const int nst = Smem::RING / stage_bytes;          // 5 or 4
    const int dig_kb = nd * dp * 128;                   // bytes of one k-block of stacked digits
    const int key_begin = rank * a.keys_per_split;
    int nkb = (min(a.L, key_begin + a.keys_per_split) - key_begin + kKeys - 1) / kKeys;
    if (nkb < 0) nkb = 0;
    const int own = (dp + cs - 1) / cs;                 // rows of W^T owned per CTA
    const int q_begin = rank * a.ra_q_per_cta;
    int nqt = (min(a.L, q_begin + a.ra_q_per_cta) - q_begin + kQTile - 1) / kQTile;
    if (nqt < 0) nqt = 0;

    if (threadIdx.x == 0) bar.init();
    if (warp == kIssuerWarp) {
        tmem_alloc(bar.tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *bar.tmem_slot;
    pdl_wait();   // packed operands come from the kernel launched just before

    bool ok = true;
    int issued = 0;                                     // producer: loads issued (both phases)
    int p_st = 0, p_round = 0;                          // producer ring position
    int c_st = 0, c_round = 0;                          // issuer ring position

    // ---------------------------------------------------------------- phase 1
    if (warp == kProducerWarp) {
        if (lane == 0) {
            tma_prefetch(&a.tm_q);
            tma_prefetch(&a.tm_k);
            tma_prefetch(&a.tm_vt);
            for (int b = 0; b < nkb; ++b) {
                if (p_round > 0 &&
                    !mbar_wait(&bar.empty[p_st], uint32_t((p_round - 1) & 1), bar.abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                uint8_t *dst = ring + p_st * stage_bytes;
                const int key0 = key_begin + b * kKeys;
                mbar_expect_tx(&bar.full[p_st], stage_bytes);
                tma_load_3d(dst, &a.tm_vt, &bar.full[p_st], key0, 0, hd);
                tma_load_3d(dst + Smem::V_TILE, &a.tm_k, &bar.full[p_st], key0, 0, hd);
                ++issued;
                if (++p_st == nst) {
                    p_st = 0;
                    ++p_round;
                }
            }
        }
    } else if (warp == kIssuerWarp) {
        const uint32_t idesc1 = make_idesc(128, dp, 0);
        for (int b = 0; ok && b < nkb; ++b) {
            if (!mbar_wait_warp(&bar.full[c_st], uint32_t(c_round & 1), bar.abort_flag, a.err)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint64_t vdesc = make_sdesc(smem_addr(ring + c_st * stage_bytes));
            const uint64_t kdesc = make_sdesc(smem_addr(ring + c_st * stage_bytes + Smem::V_TILE));
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
                mma_f16_elect(tmem, vdesc + uint64_t(kk * 2), kdesc + uint64_t(kk * 2), idesc1,
                              (b > 0 || kk > 0) ? 1u : 0u);
            tc_commit_elect(&bar.empty[c_st]);
            if (++c_st == nst) {
                c_st = 0;
                ++c_round;
            }
        }
        tc_commit_elect(bar.d1_full);                   // also fires when no MMA was issued
    }

    // ------------------------------------------- reduce W^T over the cluster
    // Drain warp w takes TMEM lane quarter w mod 4 (row j of W^T) and column
    // half (w - 2) / 4 of the partial; it waits for phase 1 before the
    // cluster barrier, after which every ring is idle and may receive rows.
    const int quarter = warp & 3;
    const int j = quarter * 32 + lane;                  // TMEM lane = row of W^T
    const int colh = (warp - 2) >> 2;
    const uint32_t lane_off = uint32_t(quarter * 32) << 16;
    uint32_t part[64];                                  // dp / 2 columns of row j
    if (warp >= 2) {
        const bool have = mbar_wait(bar.d1_full, 0, bar.abort_flag, a.err) && nkb > 0;
        if (have) tc_fence_after();
#pragma unroll
        for (int c = 0; c < 64; c += 32) {
            if (c < dp / 2) {
                uint32_t v[32];
                if (have) {
                    tmem_ld32(tmem + lane_off + uint32_t(colh * (dp / 2) + c), v);
                    tmem_wait_ld(v);
                }
#pragma unroll
                for (int x = 0; x < 32; ++x)
                    part[c + x] = have ? uint32_t(__float2int_rn(__uint_as_float(v[x]))) : 0u;
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();                                     // every CTA is past phase 1
    if (warp >= 2 && j < dp) {
        // row j -> receive buffer of its owner, slot [this rank][j - owner's first row]
        const int owner = j / own;
        const uint32_t dst = cluster_map(smem_addr(recv), uint32_t(owner)) +
                             uint32_t(((rank * own) + (j - owner * own)) * pitch + colh * (dp / 2)) * 4u;
#pragma unroll
        for (int c = 0; c < 64; c += 4)
            if (c < dp / 2) st_cluster_v4(dst + uint32_t(c) * 4u, make_uint4(part[c], part[c + 1], part[c + 2], part[c + 3]));
    }
    cluster_sync();                                     // every partial row has arrived
    if (warp >= 2) {
        // owner: rows [rank own, rank own + own) of W^T, 8 columns per item
        const int j0 = rank * own;
        const int nrows = max(0, min(own, dp - j0));
        const int sft = a.s_shift > 0 ? a.s_shift : 1;   // one digit: unused
        const int half = 1 << (sft - 1);
        const int mask = (1 << sft) - 1;
        uint32_t peer_dig[8];
#pragma unroll
        for (int r = 0; r < 8; ++r) peer_dig[r] = r < cs ? cluster_map(smem_addr(dig), uint32_t(r)) : 0u;
        for (int item = threadIdx.x - 64; item < nrows * (dp / 8); item += kDrainWarps * 32) {
            const int jj = item / (dp / 8);
            const int i0 = 8 * (item - jj * (dp / 8));
            uint32_t w[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, 0u};
            for (int src = 0; src < cs; ++src) {
                const int32_t *row = recv + (src * own + jj) * pitch + i0;
                const uint4 lo = *reinterpret_cast<const uint4 *>(row);
                const uint4 hi = *reinterpret_cast<const uint4 *>(row + 4);
                w[0] += lo.x; w[1] += lo.y; w[2] += lo.z; w[3] += lo.w;
                w[4] += hi.x; w[5] += hi.y; w[6] += hi.z; w[7] += hi.w;
            }
            // balanced digits (the plan keeps |W| < 2^31); one 16-byte chunk
            // of each digit row, stored into every CTA of the cluster
            const int kb = i0 >> 6;
            const int chunk = (i0 & 63) >> 3;
            int32_t rest[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) rest[e] = int32_t(w[e]);
            for (int dg = 0; dg < nd; ++dg) {
                __align__(16) __half h[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    int32_t v = rest[e];
                    if (dg + 1 < nd) {
                        v = ((rest[e] + half) & mask) - half;
                        rest[e] = (rest[e] - v) >> sft;
                    }
                    h[e] = __int2half_rn(v);
                }
                const int drow = dg * dp + j0 + jj;     // digits stacked along N
                const uint32_t off = uint32_t(kb * dig_kb + drow * 128 + ((chunk ^ (drow & 7)) << 4));
                const uint4 hv = *reinterpret_cast<const uint4 *>(h);
#pragma unroll
                for (int r = 0; r < 8; ++r)
                    if (r < cs) st_cluster_v4(peer_dig[r] + off, hv);
            }
        }
        // generic-proxy stores -> the tensor cores that read them as B
        asm volatile("fence.proxy.async.shared::cluster;" ::: "memory");
    }
    cluster_sync();                                     // digits complete everywhere; receive buffers read

    // ---------------------------------------------------------------- phase 2
    if (warp == kProducerWarp) {
        if (lane == 0 && ok) {
            for (int t = 0; t < nqt; ++t) {
                if (p_round > 0 &&
                    !mbar_wait(&bar.empty[p_st], uint32_t((p_round - 1) & 1), bar.abort_flag, a.err)) {
                    ok = false;
                    break;
                }
                uint8_t *dst = ring + p_st * stage_bytes;
                mbar_expect_tx(&bar.full[p_st], dkb * kQTile * 128);
                for (int kb = 0; kb < dkb; ++kb)
                    tma_load_3d(dst + kb * kQTile * 128, &a.tm_q, &bar.full[p_st], kb * 64,
                                q_begin + t * kQTile, hd);
                ++issued;
                if (++p_st == nst) {
                    p_st = 0;
                    ++p_round;
                }
            }
        }
        if (lane == 0 && *bar.abort_flag) {
            // every copy already issued lands before shared memory goes
            for (int st = 0; st < nst; ++st) {
                const int uses = issued / nst + (st < issued % nst ? 1 : 0);
                if (uses > 0) mbar_wait_drain(&bar.full[st], uint32_t((uses - 1) & 1));
            }
        }
    } else if (warp == kIssuerWarp) {
        const uint32_t idesc2 = make_idesc(128, nd * dp, 0);
        const uint64_t ddesc = make_sdesc(smem_addr(dig));
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        for (int t = 0; ok && t < nqt; ++t) {
            const int buf = t & 1;
            if (t >= 2 &&
                !mbar_wait_warp(&bar.acc_empty[buf], uint32_t(((t - 2) >> 1) & 1), bar.abort_flag, a.err)) {
                ok = false;
                break;
            }
            if (!mbar_wait_warp(&bar.full[c_st], uint32_t(c_round & 1), bar.abort_flag, a.err)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint64_t qdesc = make_sdesc(smem_addr(ring + c_st * stage_bytes));
            const uint32_t td = tmem + uint32_t(buf * 256);
            for (int kb = 0; kb < dkb; ++kb)
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)
                    mma_f16_elect(td, qdesc + uint64_t((kb * kQTile * 128 + kk * 32) >> 4),
                                  ddesc + uint64_t((kb * dig_kb + kk * 32) >> 4), idesc2,
                                  (kb > 0 || kk > 0) ? 1u : 0u);
            tc_commit_elect(&bar.empty[c_st]);
            tc_commit_elect(&bar.acc_full[buf]);
            if (++c_st == nst) {
                c_st = 0;
                ++c_round;
            }
        }
        if (!ok) {
            // MMAs already issued finish before TMEM and shared memory go
            tc_commit_elect(bar.tail);
            mbar_wait_drain(bar.tail, 0);
        }
    } else {
        // drain warps: O rows = sum_t D_t << (t s); warp w takes lane quarter
        // w mod 4 and column half (w - 2) / 4
        const int row = quarter * 32 + lane;
        const bool vec = (a.d & 3) == 0;
        const int cbeg = colh * (dp / 2);
        const int cend = min(a.d, cbeg + dp / 2);
        for (int t = 0; t < nqt; ++t) {
            const int buf = t & 1;
            const bool have = mbar_wait(&bar.acc_full[buf], uint32_t((t >> 1) & 1), bar.abort_flag, a.err);
            if (have) tc_fence_after();
            const int q = q_begin + t * kQTile + row;
            int32_t *orow = static_cast<int32_t *>(a.out) + (int64_t(hd) * a.L + q) * a.d;
            for (int c0 = cbeg; c0 < cend; c0 += 32) {
                uint32_t acc[32];
#pragma unroll
                for (int x = 0; x < 32; ++x) acc[x] = 0u;
                for (int dg = 0; have && dg < nd; ++dg) {
                    uint32_t v[32];
                    tmem_ld32(tmem + lane_off + uint32_t(buf * 256 + dg * dp + c0), v);
                    tmem_wait_ld(v);
                    const int sh = dg * a.s_shift;
                    if (a.ra_fast_cvt) {
                        // |D| < 2^22: adding 1.5 * 2^23 puts the integer in the low mantissa bits
#pragma unroll
                        for (int x = 0; x < 32; ++x)
                            acc[x] += uint32_t(__float_as_int(__uint_as_float(v[x]) + 12582912.0f) - 0x4B400000) << sh;
                    } else {
#pragma unroll
                        for (int x = 0; x < 32; ++x)
                            acc[x] += uint32_t(__float2int_rn(__uint_as_float(v[x]))) << sh;
                    }
                }
                if (q < a.L) {
#pragma unroll
                    for (int x = 0; x < 32; x += 4) {
                        const int c = c0 + x;
                        if (vec && c + 3 < a.d) {
                            *reinterpret_cast<uint4 *>(orow + c) = make_uint4(acc[x], acc[x + 1], acc[x + 2], acc[x + 3]);
                        } else {
                            if (c < a.d) orow[c] = int32_t(acc[x]);
                            if (c + 1 < a.d) orow[c + 1] = int32_t(acc[x + 1]);
                            if (c + 2 < a.d) orow[c + 2] = int32_t(acc[x + 2]);
                            if (c + 3 < a.d) orow[c + 3] = int32_t(acc[x + 3]);
                        }
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&bar.acc_empty[buf]);
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kIssuerWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ------------------------------------------------------------------- host
cudaError_t attn_reassoc_prepare() {
    return cudaFuncSetAttribute(attn_reassoc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                ra::Smem::total);
}

cudaError_t attn_reassoc_launch(const AttnArgs &a, cudaStream_t stream) {
    return launch_pdl(attn_reassoc_kernel, dim3(a.key_splits, a.heads), ra::kThreads, ra::Smem::total,
                      stream, a, a.key_splits);
}

}  // namespace qx
