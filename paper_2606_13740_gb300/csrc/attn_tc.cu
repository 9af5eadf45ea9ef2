// Bidirectional attention of the window's queries over the cached prefix and the window
// (Sec. 2.1 block-wise decoding with prefix KV reuse; no causal mask) on the 5th-generation
// tensor cores, head dim 128.
//
// One CTA = one (sequence, head, query tile of up to 128 rows) and one share of its keys; the
// csize CTAs of a cluster split the keys and merge through distributed shared memory.  Per
// 64-key sub-block j:
//   S_j = Q K_j^T         tcgen05.mma, A = Q (shared memory, K-major), B = K_j (shared,
//                         K-major), fp32 S_j in tensor memory (128 lanes = query rows)
//   P_j = exp2(S_j - m)   one thread per query row, straight from TMEM; P_j (bf16) written
//                         back into the same TMEM columns
//   O  += P_j V_j         tcgen05.mma, A = P_j from tensor memory, B = V_j (shared memory,
//                         MN-major: V is stored key-major with the head dim contiguous)
// The running max m only moves when a sub-block's max exceeds it by more than 8 (log2 units),
// and only then are O and the row sum rescaled, so P stays below 2^8 and the common case reads
// no O.  Warps 0-3: softmax and output (warp w owns TMEM lanes 32w..32w+31); warp 4: TMA loads
// and TMEM allocation; warp 5: MMA issue.  K and V have their own stages, so the next K loads
// while the current softmax and P.V run, and the next S is issued before the current P.V.
#include "common.cuh"
#include "internal.h"

namespace dllm {

namespace {

constexpr int kTcKeys = 64;          // keys per sub-block (UMMA N of Q.K^T, K of P.V)
constexpr int kTcRows = 128;         // query rows per CTA (UMMA M), padded
constexpr int kTcThreads = 192;
constexpr int kTcMaxCluster = 8;
constexpr uint32_t kTcQBytes = kTcRows * 128 * 2;   // Q tile: two 64-column halves of 16 KB
constexpr uint32_t kTcKVBytes = kTcKeys * 128 * 2;  // one K or V sub-block: two halves of 8 KB
enum { kTcStart = 0, kTcDepWait = 1, kTcLoop = 2, kTcTicket = 3, kTcMerged = 4, kTcSm = 5, kTcLast = 6,
       kTcMergeLoop = 7 };

__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
    d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
    d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
    d |= static_cast<uint64_t>(1u) << 46;  // descriptor version for tcgen05
    d |= static_cast<uint64_t>(2u) << 61;  // 128-byte swizzle
    return d;
}

// D (+)= A * B with A read from tensor memory (element (m, k) at lane m, column k/2, the even
// k in the low half), B from shared memory.
__device__ __forceinline__ void umma_tmem_a(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
        "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void tmem_st_32x32u(uint32_t taddr, const uint32_t* r) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]),
        "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]),
        "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]),
        "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void cluster_sync_tc() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t dsmem_map_tc(uint32_t saddr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
    return r;
}
__device__ __forceinline__ float2 dsmem_ld2_tc(uint32_t addr) {
    float2 v;
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr));
    return v;
}
__device__ __forceinline__ float4 dsmem_ld4_tc(uint32_t addr) {
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(addr));
    return v;
}
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ unsigned smid_tc() {
    unsigned r;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
    return r;
}

struct TcMaps {
    CUtensorMap q;  // [B*H*T][128]: box 64 x 128 rows
    CUtensorMap k;  // [B*Hkv*cap][128]: box 64 x 64 keys (Hkv: the cache's K/V heads)
    CUtensorMap v;
};

template <int NB>
__global__ void __launch_bounds__(kTcThreads, 1)
    k_attn_tc(const __grid_constant__ TcMaps maps, const int* __restrict__ seq_kv, __nv_bfloat16* __restrict__ out,
              int T, int H, int Hkv, int cap, int qtiles, int csize, int qx, int* status,
              unsigned long long* trace) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sQ = smem;                       // 32 KB
    uint8_t* sK = sQ + kTcQBytes;             // NB x 16 KB
    uint8_t* sV = sK + NB * kTcKVBytes;       // NB x 16 KB
    __shared__ uint64_t qbar, drain, kfull[NB], vfull[NB], kempty[NB], vempty[NB], sfull[2], pfull[2], pvdone[2];
    __shared__ uint32_t tslot;
    __shared__ int s_abort;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int cta = (blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
    unsigned long long* tr = (trace && cta < 256 && threadIdx.x == 0) ? trace + static_cast<size_t>(cta) * 16 : nullptr;
    if (tr) {
        tr[kTcStart] = global_ns();
        tr[kTcSm] = smid_tc();
        tr[kTcLast] = blockIdx.x == 0;
        tr[kTcMerged] = 0;
    }
    pdl_launch_dependents();
    const int split = blockIdx.x, h = blockIdx.y;
    const int b = blockIdx.z / qtiles, qt = blockIdx.z - b * qtiles;
    const int NK = seq_kv[b] + T - qx;  // the last qx rows are queries only
    const int nblk = (NK + kTcKeys - 1) / kTcKeys;
    const int blk0 = split * nblk / csize, blk1 = (split + 1) * nblk / csize;
    const int kbeg = blk0 * kTcKeys, kend = min(NK, blk1 * kTcKeys);
    const int nsub = blk1 - blk0;  // 64-key sub-blocks of this CTA (may be 0)
    const int q0 = qt * kTcRows;
    const int nq = min(kTcRows, T - q0);

    if (threadIdx.x == 0) {
        mbar_init(&qbar, 1);
        mbar_init(&drain, 1);
        for (int s = 0; s < NB; ++s) {
            mbar_init(&kfull[s], 1);
            mbar_init(&vfull[s], 1);
            mbar_init(&kempty[s], 1);
            mbar_init(&vempty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&sfull[s], 1);
            mbar_init(&pfull[s], 128);
            mbar_init(&pvdone[s], 1);
        }
        s_abort = 0;
        mbar_fence_init();
    }
    if (warp == 4) {
        tmem_alloc(&tslot, 256);  // O: columns 0..127; S/P buffers: 128..191, 192..255
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tslot;
    const uint32_t tO = tmem, tS0 = tmem + 128;

    if (warp == 4) {
        // ------------------------------------------------ loads
        if (lane == 0) {
            tma_prefetch_desc(&maps.q);
            tma_prefetch_desc(&maps.k);
            tma_prefetch_desc(&maps.v);
            pdl_wait();  // Q and the window's K/V come from the preceding projection
            if (tr) tr[kTcDepWait] = global_ns();
            const uint64_t pol_q = policy_evict_first(), pol_kv = policy_evict_first();
            const int qrow = (b * H + h) * T + q0;
            mbar_arrive_expect_tx(&qbar, kTcQBytes);
            tma_load_2d(sQ, &maps.q, 0, qrow, &qbar, pol_q);
            tma_load_2d(sQ + kTcQBytes / 2, &maps.q, 64, qrow, &qbar, pol_q);
            const int krow0 = (b * Hkv + (Hkv == H ? h : h / (H / Hkv))) * cap + kbeg;  // K/V head of query head h
            int kiss = 0, viss = 0;  // sub-blocks whose K, V copies were issued
            for (int j = 0; j < nsub && !s_abort; ++j) {
                const int st = j % NB;
                const uint32_t par = static_cast<uint32_t>((j / NB - 1) & 1);
                if (j >= NB && !mbar_wait(&kempty[st], par, &s_abort, status)) break;
                mbar_arrive_expect_tx(&kfull[st], kTcKVBytes);
                tma_load_2d(sK + st * kTcKVBytes, &maps.k, 0, krow0 + j * kTcKeys, &kfull[st], pol_kv);
                tma_load_2d(sK + st * kTcKVBytes + kTcKVBytes / 2, &maps.k, 64, krow0 + j * kTcKeys, &kfull[st], pol_kv);
                kiss = j + 1;
                if (j >= NB && !mbar_wait(&vempty[st], par, &s_abort, status)) break;
                mbar_arrive_expect_tx(&vfull[st], kTcKVBytes);
                tma_load_2d(sV + st * kTcKVBytes, &maps.v, 0, krow0 + j * kTcKeys, &vfull[st], pol_kv);
                tma_load_2d(sV + st * kTcKVBytes + kTcKVBytes / 2, &maps.v, 64, krow0 + j * kTcKeys, &vfull[st], pol_kv);
                viss = j + 1;
            }
            if (s_abort) {
                // let the copies in flight land before the shared memory is released (one
                // deadline for all)
                const long long t0 = spin_clock();
                while (!mbar_try_wait(&qbar, 0) && spin_clock() - t0 < kWaitLimitCycles) {
                }
                for (int j = max(0, kiss - NB); j < kiss; ++j)
                    while (!mbar_try_wait(&kfull[j % NB], static_cast<uint32_t>((j / NB) & 1)) &&
                           spin_clock() - t0 < kWaitLimitCycles) {
                    }
                for (int j = max(0, viss - NB); j < viss; ++j)
                    while (!mbar_try_wait(&vfull[j % NB], static_cast<uint32_t>((j / NB) & 1)) &&
                           spin_clock() - t0 < kWaitLimitCycles) {
                    }
            }
        }
    } else if (warp == 5) {
        // ------------------------------------------------ MMA issue
        if (lane == 0 && nsub > 0) {
            const uint32_t id_s = umma_idesc_bf16(kTcRows, kTcKeys);              // S = Q K^T
            const uint32_t id_o = umma_idesc_bf16(kTcRows, 128) | (1u << 16);    // O += P V, V MN-major
            bool ok = mbar_wait(&qbar, 0, &s_abort, status);
            auto issue_s = [&](int j) {  // S_j into buffer j % 2
                const int st = j % NB, sb = j % 2;
                if (!mbar_wait(&kfull[st], static_cast<uint32_t>((j / NB) & 1), &s_abort, status)) return false;
                // buffer sb last held P_{j-2}: its P.V must be done
                if (j >= 2 && !mbar_wait(&pvdone[sb], static_cast<uint32_t>(((j - 2) / 2) & 1), &s_abort, status))
                    return false;
                tc_fence_after();
                const uint32_t qa = smem_u32(sQ), ka = smem_u32(sK + st * kTcKVBytes);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {  // head dim 128 = 8 steps of 16
                    const uint32_t off = static_cast<uint32_t>((kk >> 2) * (kTcQBytes / 2) + (kk & 3) * 32);
                    const uint32_t offk = static_cast<uint32_t>((kk >> 2) * (kTcKVBytes / 2) + (kk & 3) * 32);
                    umma_bf16(tS0 + static_cast<uint32_t>(sb * 64), sw128_desc(qa + off, 16, 1024),
                              sw128_desc(ka + offk, 16, 1024), id_s, kk > 0 ? 1u : 0u);
                }
                umma_commit(&sfull[sb]);
                umma_commit(&kempty[st]);
                return true;
            };
            if (ok) ok = issue_s(0);
            for (int j = 0; j < nsub && ok; ++j) {
                if (j + 1 < nsub && !issue_s(j + 1)) break;
                const int st = j % NB, sb = j % 2;
                if (!mbar_wait(&vfull[st], static_cast<uint32_t>((j / NB) & 1), &s_abort, status)) break;
                if (!mbar_wait(&pfull[sb], static_cast<uint32_t>((j / 2) & 1), &s_abort, status)) break;
                tc_fence_after();
                const uint32_t va = smem_u32(sV + st * kTcKVBytes);
#pragma unroll
                for (int kk = 0; kk < 4; ++kk)  // 64 keys = 4 steps of 16: P columns kk*8, V key groups 2kk
                    umma_tmem_a(tO, tS0 + static_cast<uint32_t>(sb * 64 + kk * 8),
                                sw128_desc(va + static_cast<uint32_t>(kk * 2048), kTcKVBytes / 2, 1024), id_o,
                                (j > 0 || kk > 0) ? 1u : 0u);
                umma_commit(&pvdone[sb]);
                umma_commit(&vempty[st]);
            }
            // every MMA issued here is done before the CTA releases TMEM and shared memory
            umma_commit(&drain);
            const long long t0 = spin_clock();
            while (!mbar_try_wait(&drain, 0) && spin_clock() - t0 < kWaitLimitCycles) {
            }
        }
    } else {
        // ------------------------------------------------ softmax, output (warps 0..3)
        const int r = warp * 32 + lane;  // query row of the tile = TMEM lane
        const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
        const float sl2 = 0.08838834764831845f * 1.4426950408889634f;  // 1/sqrt(128) * log2(e)
        float m = -INFINITY, l = 0.0f;
        float v[64];
        bool ok = true;
        // a warp whose rows are all past the window's queries (the tile's padding) keeps step with
        // the sub-blocks but computes nothing: its rows of P and O are never read
        const bool live = warp * 32 < nq;
        for (int j = 0; j < nsub && ok; ++j) {
            const int sb = j % 2;
            ok = __all_sync(0xffffffffu, mbar_wait(&sfull[sb], static_cast<uint32_t>((j / 2) & 1), &s_abort, status));
            if (!ok) break;
            if (!live) {
                mbar_arrive(&pfull[sb]);
                continue;
            }
            tc_fence_after();
            const uint32_t ts = tS0 + static_cast<uint32_t>(sb * 64) + lane_off;
            tmem_ld_32x32(ts, v);
            tmem_ld_32x32(ts + 32, v + 32);
            const int k0 = kbeg + j * kTcKeys;
            float mx = -INFINITY;
#pragma unroll
            for (int i = 0; i < 64; ++i) {
                v[i] = (k0 + i < kend) ? v[i] * sl2 : -INFINITY;
                mx = fmaxf(mx, v[i]);
            }
            // the first sub-block, or a row max 2^8 above the one in use somewhere in the warp
            // (the whole warp rescales: TMEM accesses are warp-wide)
            if (__any_sync(0xffffffffu, mx > m + 8.0f)) {
                const float mn = fmaxf(m, mx);
                if (j > 0) {
                    // O holds P.V up to j-1: wait for the last of them, rescale O and l
                    ok = __all_sync(0xffffffffu, mbar_wait(&pvdone[(j - 1) % 2],
                                                           static_cast<uint32_t>(((j - 1) / 2) & 1), &s_abort, status));
                    if (!ok) break;
                    tc_fence_after();
                    const float al = exp2f(m - mn);
                    float o[32];
#pragma unroll 1
                    for (int c = 0; c < 128; c += 32) {
                        tmem_ld_32x32(tO + lane_off + static_cast<uint32_t>(c), o);
#pragma unroll
                        for (int i = 0; i < 32; ++i) o[i] *= al;
                        tmem_st_32x32(tO + lane_off + static_cast<uint32_t>(c), o);
                    }
                    l *= al;
                }
                m = mn;
            }
            uint32_t pk[32];
            float ls = 0.0f;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                const float p0 = exp2f(v[2 * i] - m), p1 = exp2f(v[2 * i + 1] - m);
                ls += p0 + p1;
                __nv_bfloat162 pp = __floats2bfloat162_rn(p0, p1);
                pk[i] = *reinterpret_cast<uint32_t*>(&pp);
            }
            l += ls;
            tmem_st_32x32u(ts, pk);  // P_j over the first 32 columns of the buffer
            tc_fence_before();
            mbar_arrive(&pfull[sb]);
        }
        // the output: O after the last P.V
        if (ok && nsub > 0) {
            ok = __all_sync(0xffffffffu, mbar_wait(&pvdone[(nsub - 1) % 2], static_cast<uint32_t>(((nsub - 1) / 2) & 1),
                                                   &s_abort, status));
            tc_fence_after();
        }
        if (tr && threadIdx.x == 0) tr[kTcLoop] = global_ns();
        if (!ok) l = 0.0f;
        const int qd = H * 128;
        if (csize == 1) {
            // normalised output straight from TMEM, 16-byte stores per row
            const float il = (nsub > 0 && l > 0.0f) ? 1.0f / l : 0.0f;
            __nv_bfloat16* op = out + (static_cast<size_t>(b) * T + q0 + min(r, nq - 1)) * qd + h * 128;
#pragma unroll 1
            for (int c = 0; c < 128; c += 32) {
                float o[32];
                if (nsub > 0) {
                    tmem_ld_32x32(tO + lane_off + static_cast<uint32_t>(c), o);  // all lanes: .sync.aligned
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[i] = 0.0f;
                }
                if (r < nq) {
                    uint4* dst = reinterpret_cast<uint4*>(op + c);
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        uint4 w;
                        w.x = pack_bf16x2(o[8 * i] * il, o[8 * i + 1] * il);
                        w.y = pack_bf16x2(o[8 * i + 2] * il, o[8 * i + 3] * il);
                        w.z = pack_bf16x2(o[8 * i + 4] * il, o[8 * i + 5] * il);
                        w.w = pack_bf16x2(o[8 * i + 6] * il, o[8 * i + 7] * il);
                        dst[i] = w;
                    }
                }
            }
        } else {
            // the partial (unnormalised O, max, sum) of rows < nq into shared memory, over the
            // Q/K/V tiles: every copy into them has landed and every MMA reading them is done
            // (the P.V above was the last, and MMAs complete in issue order)
            float* sO = reinterpret_cast<float*>(smem);  // [128][128]
            float* sML = sO + kTcRows * 128;             // [128][2]
#pragma unroll 1
            for (int c = 0; c < 128; c += 32) {
                float o[32];
                if (nsub > 0) {
                    tmem_ld_32x32(tO + lane_off + static_cast<uint32_t>(c), o);
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[i] = 0.0f;
                }
                if (r < nq) {
                    float4* dst = reinterpret_cast<float4*>(sO + r * 128 + c);
#pragma unroll
                    for (int i = 0; i < 8; ++i) dst[i] = make_float4(o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
                }
            }
            if (r < nq) *reinterpret_cast<float2*>(sML + r * 2) = make_float2(nsub > 0 ? m : -INFINITY, l);
        }
    }
    __syncwarp();  // the role warps reconverge before the warp-wide barriers below
    if (csize > 1) {
        cluster_sync_tc();  // every split's partial is in place
        if (tr) tr[kTcTicket] = global_ns();
        // This CTA merges output elements e = split * 192 + threadIdx.x (+ k * csize * 192): row
        // e / 32, features 4 (e % 32) .. +3, over the csize partials in CTA order.  A row is one
        // warp; lane k reads partial k's (max, sum) and the weights travel by shuffles.
        const float* sO = reinterpret_cast<const float*>(smem);
        const float* sML = sO + kTcRows * 128;
        uint32_t pb[kTcMaxCluster];
#pragma unroll
        for (int c = 0; c < kTcMaxCluster; ++c) pb[c] = c < csize ? dsmem_map_tc(smem_u32(sO), c) : 0u;
        const int nel = nq * 32;
        const int qd = H * 128;
        for (int ew0 = split * kTcThreads + warp * 32; ew0 < nel; ew0 += csize * kTcThreads) {
            const int rr = ew0 / 32, i4 = lane;  // one row per warp pass
            float mk = -INFINITY, lk = 0.0f;
            if (lane < csize) {
                const float2 ml = dsmem_ld2_tc(dsmem_map_tc(smem_u32(sML + rr * 2), static_cast<uint32_t>(lane)));
                mk = ml.x;
                lk = ml.y;
            }
            float4 ov[kTcMaxCluster];
#pragma unroll
            for (int c = 0; c < kTcMaxCluster; ++c)
                if (c < csize) ov[c] = dsmem_ld4_tc(pb[c] + static_cast<uint32_t>((rr * 128 + i4 * 4) * 4));
            float M = mk;
            M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 1));
            M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 2));
            M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 4));
            M = __shfl_sync(0xffffffffu, M, 0);
            const float wk = mk == -INFINITY ? 0.0f : exp2f(mk - M);  // a share without keys: 0
            float L = wk * lk;
            L += __shfl_xor_sync(0xffffffffu, L, 1);
            L += __shfl_xor_sync(0xffffffffu, L, 2);
            L += __shfl_xor_sync(0xffffffffu, L, 4);
            L = __shfl_sync(0xffffffffu, L, 0);
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int c = 0; c < kTcMaxCluster; ++c) {
                if (c < csize) {
                    const float w = __shfl_sync(0xffffffffu, wk, c);
                    acc.x += w * ov[c].x;
                    acc.y += w * ov[c].y;
                    acc.z += w * ov[c].z;
                    acc.w += w * ov[c].w;
                }
            }
            const float inv = L > 0.0f ? 1.0f / L : 0.0f;
            __nv_bfloat16* op = out + (static_cast<size_t>(b) * T + q0 + rr) * qd + h * 128 + i4 * 4;
            uint2 w2;
            w2.x = pack_bf16x2(acc.x * inv, acc.y * inv);
            w2.y = pack_bf16x2(acc.z * inv, acc.w * inv);
            *reinterpret_cast<uint2*>(op) = w2;
        }
        if (tr) tr[kTcMergeLoop] = global_ns();
        cluster_sync_tc();  // no CTA leaves while its partial may still be read
        if (tr) tr[kTcMerged] = global_ns();
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 4) tmem_dealloc(tmem, 256);
}

template <int NB>
size_t tc_smem() {
    return 1024 + kTcQBytes + 2 * NB * kTcKVBytes + (NB == 1 ? 1024 : 0);  // NB = 1: room for (max, sum)
}

template <int NB>
cudaError_t tc_go(cudaLaunchConfig_t& cfg, const TcMaps& maps, const int* seq_kv, __nv_bfloat16* out, int T, int H,
                  int Hkv, int cap, const AttnPlan& a, int* status, unsigned long long* trace) {
    cfg.blockDim = dim3(kTcThreads);
    cfg.dynamicSmemBytes = tc_smem<NB>();
    return cudaLaunchKernelEx(&cfg, k_attn_tc<NB>, maps, seq_kv, out, T, H, Hkv, cap, a.qtiles, a.csize, a.qx, status,
                              trace);
}

}  // namespace

cudaError_t attn_tc_init_attrs() {
    cudaError_t e = cudaFuncSetAttribute(reinterpret_cast<const void*>(k_attn_tc<1>),
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(tc_smem<1>()));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(reinterpret_cast<const void*>(k_attn_tc<2>), cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(tc_smem<2>()));
    return e;
}

AttnPlan attn_plan_tc(int B, int T, int H, int max_keys, int sms) {
    AttnPlan a{};
    a.tc = true;
    a.qtiles = (T + kTcRows - 1) / kTcRows;
    const int units = B * H * a.qtiles;
    const int blocks = (max_keys + kTcKeys - 1) / kTcKeys;
    // key splits (cluster size): about two CTAs per SM, at most one split per sub-block
    int c = (2 * sms + units - 1) / units;
    if (c > kTcMaxCluster) c = kTcMaxCluster;
    if (c > blocks) c = blocks;
    if (c < 1) c = 1;
    a.csize = c;
    a.nb = (blocks + c - 1) / c >= 3 ? 2 : 1;  // long key ranges keep two K/V sub-blocks in flight
    return a;
}

cudaError_t launch_attention_tc(const __nv_bfloat16* q, const __nv_bfloat16* kc, const __nv_bfloat16* vc,
                                const int* seq_kv, __nv_bfloat16* out, int B, int T, int H, int Hkv, int cap,
                                const AttnPlan& a, cudaStream_t st, bool pdl, unsigned long long* trace,
                                int* status) {
    if (a.csize < 1 || a.csize > kTcMaxCluster || (a.nb != 1 && a.nb != 2) || Hkv < 1 || H % Hkv)
        return cudaErrorInvalidValue;
    TcMaps maps;
    if (!make_tmap_bf16(&maps.q, q, static_cast<uint64_t>(B) * H * T, 128, kTcRows) ||
        !make_tmap_bf16(&maps.k, kc, static_cast<uint64_t>(B) * Hkv * cap, 128, kTcKeys) ||
        !make_tmap_bf16(&maps.v, vc, static_cast<uint64_t>(B) * Hkv * cap, 128, kTcKeys))
        return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(a.csize, H, B * a.qtiles);
    cfg.stream = st;
    cudaLaunchAttribute at[2];
    int n = 0;
    at[n].id = cudaLaunchAttributeClusterDimension;
    at[n].val.clusterDim.x = static_cast<unsigned>(a.csize);
    at[n].val.clusterDim.y = 1;
    at[n].val.clusterDim.z = 1;
    ++n;
    if (pdl && pdl_enabled()) {
        at[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    cfg.attrs = at;
    cfg.numAttrs = n;
    return a.nb == 2 ? tc_go<2>(cfg, maps, seq_kv, out, T, H, Hkv, cap, a, status, trace)
                     : tc_go<1>(cfg, maps, seq_kv, out, T, H, Hkv, cap, a, status, trace);
}

}  // namespace dllm
