// One split of the mma.sync attention kernel (k_attn, kernels.cu): the online-softmax pass of
// one query tile (16 rows per warp) over the keys [kbeg, kend) of one (sequence, head), on bf16
// mma.sync tiles.
#pragma once

#include "common.cuh"

namespace dllm {

constexpr int kAK = 64;  // keys per sub-block

__device__ __forceinline__ int swz(int r, int c, int hd) {
    return r * hd + ((((c >> 3) ^ (r & 7))) << 3) + (c & 7);
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
    unsigned s = smem_u32(dst);
    int n = valid ? 16 : 0;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(s), "l"(src), "r"(n) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { cp_async_wait<0>(); }
__device__ __forceinline__ void cp_async_wait_1() { cp_async_wait<1>(); }

__device__ __forceinline__ void ldm_x4(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c, uint32_t& d) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
                 : "r"(addr));
}
__device__ __forceinline__ void ldm_x4_t(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c, uint32_t& d) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
                 : "r"(addr));
}
__device__ __forceinline__ void mma16816(float* d, uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}


// Issues the copies of the first K and V sub-block when it lies entirely in the cached prefix
// (no earlier kernel writes it, so this may precede the dependency wait).  Returns whether it
// did (the cp.async group order attn_split expects).  NT threads, tid in [0, NT).
template <int HD, int NT>
__device__ __forceinline__ bool attn_prefetch_prefix(const __nv_bfloat16* kbase, const __nv_bfloat16* vbase, int kv,
                                                     int kbeg, int kend, __nv_bfloat16* sK, __nv_bfloat16* sV,
                                                     int tid) {
    constexpr int CPR = HD / 8;  // 16-byte chunks per row
    const bool prefix_first = kbeg < kend && kbeg + kAK <= kv;
    if (prefix_first) {  // groups: K0, V0 (then Q)
        for (int e = tid; e < kAK * CPR; e += NT) {
            const int r = e / CPR, cc = (e % CPR) * 8;
            cp_async16(sK + swz(r, cc, HD), kbase + static_cast<size_t>(kbeg + r) * HD + cc, true);
        }
        cp_async_commit();
        for (int e = tid; e < kAK * CPR; e += NT) {
            const int r = e / CPR, cc = (e % CPR) * 8;
            cp_async16(sV + swz(r, cc, HD), vbase + static_cast<size_t>(kbeg + r) * HD + cc, true);
        }
        cp_async_commit();
    }
    return prefix_first;
}

// The split proper (after the dependency wait): NW warps, tid in [0, 32 NW), nq valid query
// rows of the tile at qbase; shared Q [16 NW][HD], K and V [NB][kAK][HD]; sync() synchronises
// the NW warps.  NB = 1: the next sub-block's K streams in behind this one's softmax and P.V,
// its V behind the next Q.K^T; NB = 2 (long key ranges): two sub-blocks ahead.  Out: unnormalised o for rows r0 = 16 warp + lane/4 and r1 = r0 + 8
// (columns dn*8 + 2 (lane%4) + {0,1}), their running max (log2 units) and sum.  A split
// without keys leaves o = 0, m = -inf, l = 0.
template <int HD, int NW, int NB, typename Sync>
__device__ __forceinline__ void attn_split(const __nv_bfloat16* qbase, const __nv_bfloat16* kbase,
                                           const __nv_bfloat16* vbase, int kbeg, int kend, int nq, bool prefix_first,
                                           __nv_bfloat16* sQ, __nv_bfloat16* sK, __nv_bfloat16* sV, int tid, Sync sync,
                                           float (&o)[HD / 8][4], float& m0, float& m1, float& l0, float& l1) {
    constexpr int AQ = NW * 16;
    constexpr int NT = NW * 32;
    constexpr int CPR = HD / 8;  // 16-byte chunks per row
    const int warp = tid >> 5, lane = tid & 31;
    const int c4 = lane & 3;
    auto load_rows = [&](__nv_bfloat16* dst, const __nv_bfloat16* base, int k0) {
        for (int e = tid; e < kAK * CPR; e += NT) {
            const int r = e / CPR, cc = (e % CPR) * 8;
            const int key = k0 + r;
            const bool ok = key < kend;
            cp_async16(dst + swz(r, cc, HD), base + static_cast<size_t>(ok ? key : kbeg) * HD + cc, ok);
        }
    };
    const bool has = kbeg < kend;
    for (int e = tid; e < AQ * CPR; e += NT) {
        const int r = e / CPR, cc = (e % CPR) * 8;
        cp_async16(sQ + swz(r, cc, HD), qbase + static_cast<size_t>(r < nq ? r : 0) * HD + cc, r < nq);
    }
    if (has && !prefix_first) load_rows(sK, kbase, kbeg);
    cp_async_commit();  // group: Q (+ K0)
    if (has && !prefix_first) {
        load_rows(sV, vbase, kbeg);
        cp_async_commit();  // group: V0
    }
    if constexpr (NB == 2) {
        // groups so far: K0, V0, Q (prefix first) or Q+K0, V0; then K1, V1 (empty past the end)
        if (kbeg + kAK < kend) load_rows(sK + kAK * HD, kbase, kbeg + kAK);
        cp_async_commit();
        if (kbeg + kAK < kend) load_rows(sV + kAK * HD, vbase, kbeg + kAK);
        cp_async_commit();
    }

    constexpr int KS = HD / 16;  // k-steps of Q.K
    constexpr int DN = HD / 8;   // output n-blocks
    uint32_t qa[KS][4];
#pragma unroll
    for (int i = 0; i < DN; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.0f;
    m0 = -INFINITY;
    m1 = -INFINITY;
    l0 = 0.0f;
    l1 = 0.0f;
    const float sl2 = rsqrtf(static_cast<float>(HD)) * 1.4426950408889634f;

    int it = 0;
    for (int k0 = kbeg; k0 < kend; k0 += kAK, ++it) {
        const bool first = k0 == kbeg;
        const bool more = k0 + kAK < kend;
        __nv_bfloat16* K = sK + (NB == 2 ? (it & 1) * kAK * HD : 0);
        __nv_bfloat16* V = sV + (NB == 2 ? (it & 1) * kAK * HD : 0);
        if constexpr (NB == 1) {
            // pending groups, oldest first: K_i, V_i (first: K0, V0, Q or Q+K0, V0)
            if (first && prefix_first) cp_async_wait_all();
            else cp_async_wait_1();
        } else {
            // the three most recent groups may stay pending (V_i, K_i+1, V_i+1; first sub-block
            // with the prefix fetched early: K1, V1 after Q)
            if (first && prefix_first) cp_async_wait<2>();
            else cp_async_wait<3>();
        }
        sync();
        if (first) {
#pragma unroll
            for (int ks = 0; ks < KS; ++ks) {
                const int r = warp * 16 + (lane & 15), cc = ks * 16 + (lane >> 4) * 8;
                ldm_x4(smem_u32(sQ + swz(r, cc, HD)), qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3]);
            }
        }
        float s[8][4];
#pragma unroll
        for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.0f;
#pragma unroll
        for (int jp = 0; jp < 4; ++jp) {
#pragma unroll
            for (int ks = 0; ks < KS; ++ks) {
                const int mi = lane >> 3, rr = lane & 7;
                const int key = jp * 16 + (mi >> 1) * 8 + rr, cc = ks * 16 + (mi & 1) * 8;
                uint32_t b0, b1, b2, b3;
                ldm_x4(smem_u32(K + swz(key, cc, HD)), b0, b1, b2, b3);
                mma16816(s[2 * jp], qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], b0, b1);
                mma16816(s[2 * jp + 1], qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], b2, b3);
            }
        }
        sync();  // K consumed: the next sub-block's K streams in behind the softmax and P.V
        if constexpr (NB == 1) {
            if (more) {
                load_rows(sK, kbase, k0 + kAK);
                cp_async_commit();
            }
        } else {  // K two sub-blocks ahead into the buffer just read (an empty group past the end)
            if (k0 + 2 * kAK < kend) load_rows(K, kbase, k0 + 2 * kAK);
            cp_async_commit();
        }
        // scale to log2 units, mask keys past the end, online softmax
        float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int key = k0 + j * 8 + 2 * c4;
            const bool v0 = key < kend, v1 = key + 1 < kend;
            s[j][0] = v0 ? s[j][0] * sl2 : -INFINITY;
            s[j][1] = v1 ? s[j][1] * sl2 : -INFINITY;
            s[j][2] = v0 ? s[j][2] * sl2 : -INFINITY;
            s[j][3] = v1 ? s[j][3] * sl2 : -INFINITY;
            mx0 = fmaxf(mx0, fmaxf(s[j][0], s[j][1]));
            mx1 = fmaxf(mx1, fmaxf(s[j][2], s[j][3]));
        }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
        const float ms0 = mn0 == -INFINITY ? 0.0f : mn0, ms1 = mn1 == -INFINITY ? 0.0f : mn1;
        const float al0 = exp2f(m0 - ms0), al1 = exp2f(m1 - ms1);
        m0 = mn0;
        m1 = mn1;
        l0 *= al0;
        l1 *= al1;
#pragma unroll
        for (int i = 0; i < DN; ++i) {
            o[i][0] *= al0;
            o[i][1] *= al0;
            o[i][2] *= al1;
            o[i][3] *= al1;
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            s[j][0] = exp2f(s[j][0] - ms0);
            s[j][1] = exp2f(s[j][1] - ms0);
            s[j][2] = exp2f(s[j][2] - ms1);
            s[j][3] = exp2f(s[j][3] - ms1);
            l0 += s[j][0] + s[j][1];
            l1 += s[j][2] + s[j][3];
        }
        if constexpr (NB == 1) {
            // pending: V_i (+ K_{i+1})
            if (more) cp_async_wait_1();
            else cp_async_wait_all();
        } else {
            cp_async_wait<3>();  // V_i done; K_i+1, V_i+1, K_i+2 may stay pending
        }
        sync();
        // O += P V
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            const uint32_t a0 = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
            const uint32_t a1 = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
            const uint32_t a2 = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
            const uint32_t a3 = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
            for (int dn = 0; dn < DN; dn += 2) {
                const int mi = lane >> 3, rr = lane & 7;
                const int key = kk * 16 + (mi & 1) * 8 + rr, cc = (dn + (mi >> 1)) * 8;
                uint32_t b0, b1, b2, b3;
                ldm_x4_t(smem_u32(V + swz(key, cc, HD)), b0, b1, b2, b3);
                mma16816(o[dn], a0, a1, a2, a3, b0, b1);
                mma16816(o[dn + 1], a0, a1, a2, a3, b2, b3);
            }
        }
        sync();  // V consumed
        if constexpr (NB == 1) {
            if (more) {
                load_rows(sV, vbase, k0 + kAK);
                cp_async_commit();
            }
        } else {
            if (k0 + 2 * kAK < kend) load_rows(V, vbase, k0 + 2 * kAK);
            cp_async_commit();
        }
    }
    cp_async_wait_all();  // a CTA without keys still has its Q copy in flight
    sync();
    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);

}

}  // namespace dllm
