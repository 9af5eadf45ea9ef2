// Element-wise, normalisation, attention and bookkeeping kernels of the
// denoising step.  The dense projections live in gemm_tc.cu.
#include "attn.cuh"
#include "common.cuh"
#include "internal.h"

#include <climits>

namespace dllm {

// ------------------------------------------------------------------ weight generator
// SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): the n-th output of a stream
// whose state starts at `key` is mix(key + (n+1) * golden_gamma).
__host__ __device__ __forceinline__ uint64_t sm64_at_hd(uint64_t key, uint64_t n) {
    uint64_t z = key + (n + 1ull) * 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

// Element i of a tensor: four 32-bit draws summed (Irwin-Hall of order 4),
// centred at 2^33, scaled by sqrt(3)/2^32 to unit variance, times sigma;
// each double operation rounded once (IEEE round-to-nearest).
__device__ __forceinline__ float gen_value(uint64_t key, uint64_t i, double sigma) {
    uint64_t s = 0;
#pragma unroll
    for (uint64_t j = 0; j < 4; ++j) s += sm64_at_hd(key, 4ull * i + j) >> 32;
    double centred = __dsub_rn(__ull2double_rn(s), 8589934592.0);
    double unit = __dmul_rn(centred, 0x1.bb67ae8584caap-32);
    double scaled = __dmul_rn(unit, sigma);
    return __double2float_rn(scaled);
}

// Row map shared by the bf16 and 4-bit generators: physical row r of a fused matrix -> the
// tensor (tid0 + part) and logical row it holds (logical_rows: a padding row).
__device__ __forceinline__ void weight_row(int mode, int r, int qd, int kvd, int hd, int logical_rows, uint64_t tid0,
                                           uint64_t* tid, int* lr) {
    *tid = tid0;
    *lr = r;
    if (mode == 1) {
        const int part = r < qd ? 0 : (r < qd + kvd ? 1 : (r < qd + 2 * kvd ? 2 : 3));
        const int f = r - (part == 0 ? 0 : qd + (part - 1) * kvd);
        const int hh = f / hd, pp = f % hd;
        *tid = tid0 + part;
        *lr = hh * hd + (pp >> 1) + (pp & 1) * (hd >> 1);
        if (part > 2 || *lr >= (part == 0 ? qd : kvd)) *lr = logical_rows;
    } else if (mode == 2) {
        const int tile = r >> 7, w = r & 127;
        *tid = tid0 + (w & 1);
        *lr = tile * 64 + (w >> 1);
    }
}

// mode 0: plain (physical row = logical row of tensor tid0, zero rows past
//         logical_rows);
// mode 1: fused QKV: rows [0,qd) tensor tid0 (q), [qd,qd+kvd) tid0+1 (k), [qd+kvd,qd+2kvd)
//         tid0+2 (v) (kvd = K/V heads x hd: fewer K/V heads than query heads under grouped-query
//         attention); inside each head of hd rows, physical row 2j holds feature j and row 2j+1
//         feature j + hd/2 (the rotate-half RoPE pair sits in adjacent TMEM lanes);
// mode 2: fused gate/up: 128-row tile k, physical row 2f = gate row 64k+f (tensor tid0),
//         row 2f+1 = up row 64k+f (tensor tid0+1); zero past logical_rows.
// Storage: row-major, or tile-major (tiled_index) when tiled; the loop walks the destination in
// storage order.
__global__ void k_init_weight(__nv_bfloat16* dst, int mode, int rows, int cols, int logical_rows, uint64_t seed,
                              uint64_t tid0, int qd, int kvd, int hd, int tiled) {
    const int kb = (cols + 63) / 64;
    const size_t n = tiled ? static_cast<size_t>(rows) * kb * 64 : static_cast<size_t>(rows) * cols;
    for (size_t e = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; e < n;
         e += static_cast<size_t>(gridDim.x) * blockDim.x) {
        int r, c;
        if (tiled) {
            const size_t tile = e >> 13;
            const int w = static_cast<int>(e & 8191), rr = w >> 6;
            const int mt = static_cast<int>(tile / kb), kt = static_cast<int>(tile - static_cast<size_t>(mt) * kb);
            r = mt * 128 + rr;
            c = kt * 64 + ((((w & 63) >> 3) ^ (rr & 7)) << 3) + (w & 7);
            if (c >= cols) {
                dst[e] = __float2bfloat16_rn(0.0f);
                continue;
            }
        } else {
            r = static_cast<int>(e / cols);
            c = static_cast<int>(e - static_cast<size_t>(r) * cols);
        }
        uint64_t tid;
        int lr;
        weight_row(mode, r, qd, kvd, hd, logical_rows, tid0, &tid, &lr);
        float v = 0.0f;
        if (lr < logical_rows) {
            uint64_t key = sm64_at_hd(seed, tid);
            v = gen_value(key, static_cast<uint64_t>(lr) * cols + c, 0.02);
        }
        dst[e] = __float2bfloat16_rn(v);
    }
}

cudaError_t launch_init_weight(__nv_bfloat16* dst, int mode, int rows_phys, int cols, int logical_rows,
                               uint64_t seed, uint64_t tid0, int qd, int kvd, int hd, bool tiled, cudaStream_t st) {
    if (tiled && (rows_phys & 127)) return cudaErrorInvalidValue;
    size_t n = static_cast<size_t>(rows_phys) * (tiled ? (cols + 63) / 64 * 64 : cols);
    int blocks = static_cast<int>((n + 255) / 256 < 65536 ? (n + 255) / 256 : 65536);
    k_init_weight<<<blocks, 256, 0, st>>>(dst, mode, rows_phys, cols, logical_rows, seed, tid0, qd, kvd, hd,
                                          tiled ? 1 : 0);
    return cudaGetLastError();
}

// Seeded 4-bit block-quantised weights (the Q4_0 format of the paper's runs) in the tile layout
// of kQ4TileBytes (internal.h).  Code of logical element (lr, c) of tensor tid: the top 4 bits
// of SplitMix64 output lr * cols + c of the stream keyed by (seed, 3 * 2^40 + tid); scale of
// block (lr, b): bf16 bits 0x3B80 | the top 5 bits of output lr * ceil(cols / 32) + b of the
// stream keyed by (seed, 4 * 2^40 + tid), i.e. (1 + m/128) * 2^-8 with m < 32 (weights of
// standard deviation about 0.02).  Padding rows: scale 0; columns past cols: code 8.
// One thread per (tile, row, code word or scale).
__global__ void k_init_weight_q4(uint8_t* dst, int mode, int rows, int cols, int logical_rows, uint64_t seed,
                                 uint64_t tid0, int qd, int kvd, int hd) {
    const int kb = (cols + 63) / 64;
    const int nblk = (cols + 31) / 32;
    const size_t n = static_cast<size_t>(rows / 128) * kb * 128 * 10;
    for (size_t e = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; e < n;
         e += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const size_t tile = e / 1280;
        const int w = static_cast<int>(e - tile * 1280), rr = w & 127, item = w >> 7;
        const int mt = static_cast<int>(tile / kb), kt = static_cast<int>(tile - static_cast<size_t>(mt) * kb);
        uint64_t tid;
        int lr;
        weight_row(mode, mt * 128 + rr, qd, kvd, hd, logical_rows, tid0, &tid, &lr);
        const bool valid = lr < logical_rows;
        uint8_t* tb = dst + tile * kQ4TileBytes;
        if (item < 8) {
            const uint64_t key = sm64_at_hd(seed, (3ull << 40) + tid);
            uint32_t word = 0;
            for (int j = 0; j < 8; ++j) {
                const int c = kt * 64 + item * 8 + j;
                const uint32_t code =
                    (valid && c < cols)
                        ? static_cast<uint32_t>(sm64_at_hd(key, static_cast<uint64_t>(lr) * cols + c) >> 60)
                        : 8u;
                word |= code << q4_code_shift(j);
            }
            reinterpret_cast<uint32_t*>(tb)[item * 128 + rr] = word;
        } else {
            const int b = item - 8;
            const uint64_t key = sm64_at_hd(seed, (4ull << 40) + tid);
            const int blk = 2 * kt + b;
            const uint16_t bits =
                (valid && blk < nblk)
                    ? static_cast<uint16_t>(0x3B80u | static_cast<uint32_t>(
                                                          sm64_at_hd(key, static_cast<uint64_t>(lr) * nblk + blk) >> 59))
                    : static_cast<uint16_t>(0);
            reinterpret_cast<uint16_t*>(tb + 4096)[b * 128 + rr] = bits;
        }
    }
}

cudaError_t launch_init_weight_q4(uint8_t* dst, int mode, int rows_phys, int cols, int logical_rows, uint64_t seed,
                                  uint64_t tid0, int qd, int kvd, int hd, cudaStream_t st) {
    if (rows_phys & 127) return cudaErrorInvalidValue;
    const size_t n = static_cast<size_t>(rows_phys / 128) * ((cols + 63) / 64) * 1280;
    const int blocks = static_cast<int>((n + 255) / 256 < 65536 ? (n + 255) / 256 : 65536);
    k_init_weight_q4<<<blocks, 256, 0, st>>>(dst, mode, rows_phys, cols, logical_rows, seed, tid0, qd, kvd, hd);
    return cudaGetLastError();
}

// Synthetic prefix KV: cache[b][h][pos][i] for pos < P is element pos*(H*hd) + h*hd + i
// of tensor 2^32 + ((b*L + layer)*2 + which), sigma 1 (H: the cache's K/V heads).
__global__ void k_init_kv(__nv_bfloat16* cache, int B, int H, int hd, int cap, int P, int layer, int which, int L,
                          uint64_t seed) {
    const size_t n = static_cast<size_t>(B) * H * P * hd;
    const int qd = H * hd;
    for (size_t e = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; e < n;
         e += static_cast<size_t>(gridDim.x) * blockDim.x) {
        int i = static_cast<int>(e % hd);
        size_t r = e / hd;
        int pos = static_cast<int>(r % P);
        r /= P;
        int h = static_cast<int>(r % H);
        int b = static_cast<int>(r / H);
        uint64_t tid = 0x100000000ull + (static_cast<uint64_t>(b) * L + layer) * 2ull + which;
        uint64_t key = sm64_at_hd(seed, tid);
        float v = gen_value(key, static_cast<uint64_t>(pos) * qd + h * hd + i, 1.0);
        cache[((static_cast<size_t>(b) * H + h) * cap + pos) * hd + i] = __float2bfloat16_rn(v);
    }
}

cudaError_t launch_init_kv_random(__nv_bfloat16* cache, int B, int H, int hd, int cap, int P, int layer, int which,
                                  int L, uint64_t seed, cudaStream_t st) {
    size_t n = static_cast<size_t>(B) * H * P * hd;
    if (n == 0) return cudaSuccess;
    int blocks = static_cast<int>((n + 255) / 256 < 65536 ? (n + 255) / 256 : 65536);
    k_init_kv<<<blocks, 256, 0, st>>>(cache, B, H, hd, cap, P, layer, which, L, seed);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ embedding
// One CTA (8 warps) per token: x = embedding row (fp32 residual), xb = bf16(x)
// (the QKV projection's operand), sq[c][token] = sum of x^2 over features
// [128c, 128c+128) (the first RMSNorm's statistics, merged in the consumer),
// cur[token] = the id (for the LM head's current-token probability).
__global__ void __launch_bounds__(256) k_embed(const int* tok, int tok_ld, const int* seq_kv,
                                               const __nv_bfloat16* emb, float* x, __nv_bfloat16* xb, float* sq,
                                               int* cur, int* epoch, int T, int N, int d, int Tw, const int* trk) {
    pdl_wait();
    pdl_launch_dependents();
    const int j = blockIdx.x;
    if (j == 0 && threadIdx.x == 0) *epoch += 1;  // one forward pass: a new tag for the chained projections
    const int b = j / T, t = j - b * T;
    // window rows, then (sparse cache refresh, one sequence) the tracked prefix positions
    const int pos = t < Tw ? seq_kv[b] + t : trk[b * (T - Tw) + t - Tw];
    const int id = pos >= 0 ? tok[static_cast<size_t>(b) * tok_ld + pos] : 0;
    if (threadIdx.x == 0) cur[j] = id;
    const __nv_bfloat16* e = emb + static_cast<size_t>(id) * d;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int c = warp; c * 128 < d; c += blockDim.x >> 5) {
        float ss = 0.0f;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int i = c * 128 + r * 32 + lane;
            const __nv_bfloat16 h = e[i];
            const float v = __bfloat162float(h);
            x[static_cast<size_t>(j) * d + i] = v;
            xb[static_cast<size_t>(j) * d + i] = h;
            ss += v * v;
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ss += __shfl_down_sync(0xffffffffu, ss, off);
        if (lane == 0) sq[static_cast<size_t>(c) * N + j] = ss;
    }
}

cudaError_t launch_embed(const int* tok, int tok_ld, const int* seq_kv, const __nv_bfloat16* emb, float* x,
                         __nv_bfloat16* xb, float* sq, int* cur, int* epoch, int B, int T, int d, cudaStream_t st,
                         int Tw, const int* trk) {
    if (Tw < 0) Tw = T;
    if (Tw < T && !trk) return cudaErrorInvalidValue;
    return launch_k(k_embed, dim3(B * T), dim3(256), 0, st, true, tok, tok_ld, seq_kv, emb, x, xb, sq, cur, epoch, T,
                    B * T, d, Tw, trk);
}

// ------------------------------------------------------------------ attention
// Bidirectional attention of T window queries per sequence over keys
// [0, kv_len + T) of the KV cache (cached prefix, then the window's own keys
// written by the QKV epilogue), flash style: online softmax over 64-key
// sub-blocks on bf16 mma.sync tiles, NW warps of 16 query rows per CTA.
//
// Split-KV over a thread-block cluster: the csize CTAs of a cluster share one
// (sequence, head, query tile) and take consecutive, balanced shares of its
// key sub-blocks.  Each leaves its unnormalised output and (max, sum) per row
// in its own shared memory; after a cluster barrier every CTA merges a slice
// of the rows by reading all csize partials through distributed shared memory,
// so the merge needs no global scratch, no fences and no atomics.
constexpr int kMaxCluster = 8;
// attention timeline slots (%globaltimer ns)
enum { kAtStart = 0, kAtDepWait = 1, kAtLoop = 2, kAtTicket = 3, kAtMerged = 4, kAtSm = 5, kAtLast = 6,
       kAtMergeLoop = 7 };

__device__ __forceinline__ unsigned smid_attn() {
    unsigned r;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(r));
    return r;
}

// ---- thread-block cluster helpers
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared-memory location in CTA `rank` of this cluster.
__device__ __forceinline__ uint32_t dsmem_map(uint32_t saddr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
    return r;
}
// (no memory clobber: used only between cluster barriers, so the loads may be scheduled
// together)
__device__ __forceinline__ float2 dsmem_ld2(uint32_t addr) {
    float2 v;
    asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr));
    return v;
}
__device__ __forceinline__ float4 dsmem_ld4(uint32_t addr) {
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(addr));
    return v;
}

// Shared memory: Q tile [16*NW][HD], one K and one V sub-block [64][HD] (bf16,
// XOR-swizzled 16-byte chunks).  The next sub-block's K streams in while this
// one's softmax and P.V run, its V while the next Q.K^T runs.  After the key
// loop the same memory holds the CTA's partial: O [16*NW][HD] fp32 and
// (max, sum) [16*NW][2].
template <int HD, int NW, int NB, int PR>
__global__ void __launch_bounds__(PR * NW * 32) k_attn(const __nv_bfloat16* __restrict__ q,
                                                       const __nv_bfloat16* __restrict__ kc,
                                                       const __nv_bfloat16* __restrict__ vc,
                                                       const int* __restrict__ seq_kv, __nv_bfloat16* __restrict__ out,
                                                       int T, int H, int Hkv, int cap, int qtiles, int csize,
                                                       int qx, unsigned long long* trace, const AttnSync sy,
                                                       int* status) {
    constexpr int AQ = NW * 16;  // query rows per CTA
    constexpr int NT = NW * 32;  // threads of one warp group
    constexpr int PART = (AQ + 2 * NB * kAK) * HD * 2;  // one group's Q, K, V tiles
    extern __shared__ __align__(128) uint8_t smem_attn[];
    const int cta = (blockIdx.z * gridDim.y + blockIdx.y) * gridDim.x + blockIdx.x;
    unsigned long long* tr = (trace && cta < 256 && threadIdx.x == 0) ? trace + static_cast<size_t>(cta) * 16 : nullptr;
    if (tr) {
        tr[kAtStart] = global_ns();
        tr[kAtSm] = smid_attn();
        tr[kAtLast] = blockIdx.x == 0;
        tr[kAtMerged] = 0;
    }
    // seq_kv and the cached prefix rows are not written by the preceding kernel (the QKV
    // projection writes the window rows [kv_len, kv_len + T)), so they may be read before
    // the dependency wait
    pdl_launch_dependents();
    // PR groups of NW warps per CTA, each on its own share of the CTA's key sub-blocks
    const int grp = threadIdx.x / NT;
    __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem_attn + grp * PART);
    __nv_bfloat16* sK = sQ + AQ * HD;
    __nv_bfloat16* sV = sK + NB * kAK * HD;

    const int split = blockIdx.x, h = blockIdx.y;  // split = rank in the cluster
    const int b = blockIdx.z / qtiles, qt = blockIdx.z - b * qtiles;
    const int kv = seq_kv[b];
    const int NK = kv + T - qx;  // the last qx rows are queries only
    const int nblk = (NK + kAK - 1) / kAK;
    const int blk0 = split * nblk / csize, blk1 = (split + 1) * nblk / csize;  // the CTA's sub-blocks
    const int kbeg = (blk0 + grp * (blk1 - blk0) / PR) * kAK;
    const int kend = min(NK, (blk0 + (grp + 1) * (blk1 - blk0) / PR) * kAK);  // empty when kbeg >= kend
    const int q0 = qt * AQ;
    const int nq = min(AQ, T - q0);
    const int tid = threadIdx.x - grp * NT, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, c4 = lane & 3;

    const __nv_bfloat16* qbase = q + ((static_cast<size_t>(b) * H + h) * T + q0) * HD;
    // grouped-query attention: query head h reads K/V head h / (H / Hkv)
    const int hk = Hkv == H ? h : h / (H / Hkv);
    const __nv_bfloat16* kbase = kc + (static_cast<size_t>(b) * Hkv + hk) * cap * HD;
    const __nv_bfloat16* vbase = vc + (static_cast<size_t>(b) * Hkv + hk) * cap * HD;

    auto sync = [grp]() {
        if constexpr (PR == 1) __syncthreads();
        else named_bar(1 + grp, NT);
    };
    const bool prefix_first = attn_prefetch_prefix<HD, NT>(kbase, vbase, kv, kbeg, kend, sK, sV, tid);
    if (sy.qkv_done) {
        // the QKV tiles holding this sequence's window rows of q head h, K head hk and V head hk.
        // On a timeout the status word records it and the CTA goes on (its cluster peers wait
        // for it at the merge); the launch's result is then discarded.
        // Warp 0 polls them side by side, one flag per lane (q, K, V for each token tile).
        if (threadIdx.x < 32) {
            const int tag = *reinterpret_cast<const volatile int*>(sy.epoch) * sy.tag_mul + sy.tag_add;
            const int nt0 = (b * T) / sy.qkv_ntile, nts = (b * T + T - 1) / sy.qkv_ntile - nt0 + 1;
            const int lane = threadIdx.x;
            for (int f0 = 0; f0 < 3 * nts; f0 += 32) {
                const int fi = f0 + lane;
                const int* f = nullptr;
                if (fi < 3 * nts) {
                    const int which = fi / nts, nt = nt0 + fi - which * nts;
                    const int row = which == 0 ? h * HD : (which == 1 ? sy.k_row0 : sy.v_row0) + hk * HD;
                    f = sy.qkv_done + static_cast<size_t>(row / 128) * sy.qkv_ntiles + nt;
                }
                const long long t0 = spin_clock();
                for (;;) {
                    const bool ok = !f || ld_acquire(f) == tag;
                    if (__all_sync(0xffffffffu, ok)) break;
                    if (spin_clock() - t0 > kWaitLimitCycles) {  // warp-uniform (one clock read)
                        if (!ok && status) atomicOr(status, kStatusTimeout);
                        break;
                    }
                    __nanosleep(32);
                }
            }
        }
        __syncthreads();
    } else {
        pdl_wait();
    }
    if (tr) tr[kAtDepWait] = global_ns();
    constexpr int DN = HD / 8;  // output n-blocks
    float o[DN][4];
    float m0, m1, l0, l1;
    attn_split<HD, NW, NB>(qbase, kbase, vbase, kbeg, kend, nq, prefix_first, sQ, sK, sV, tid, sync, o, m0, m1, l0,
                           l1);
    if (tr) tr[kAtLoop] = global_ns();

    const int r0 = warp * 16 + g, r1 = r0 + 8;
    const int qd = H * HD;
    if constexpr (PR == 2) {
        // the two groups hold the same rows and columns of the tile (same warp, same lane):
        // group 1 hands its partial over through its own, finished, shared memory and group 0
        // merges it in registers, so the cluster sees one partial per CTA
        float* x = reinterpret_cast<float*>(smem_attn + PART);  // [DN*4 + 4][NT], conflict-free
        if (grp == 1) {
#pragma unroll
            for (int dn = 0; dn < DN; ++dn)
#pragma unroll
                for (int j = 0; j < 4; ++j) x[(dn * 4 + j) * NT + tid] = o[dn][j];
            x[(DN * 4 + 0) * NT + tid] = m0;
            x[(DN * 4 + 1) * NT + tid] = m1;
            x[(DN * 4 + 2) * NT + tid] = l0;
            x[(DN * 4 + 3) * NT + tid] = l1;
        }
        __syncthreads();
        if (grp == 0) {
            const float n0 = x[(DN * 4 + 0) * NT + tid], n1 = x[(DN * 4 + 1) * NT + tid];
            const float k0 = x[(DN * 4 + 2) * NT + tid], k1 = x[(DN * 4 + 3) * NT + tid];
            const float M0 = fmaxf(m0, n0), M1 = fmaxf(m1, n1);
            const float s0 = M0 == -INFINITY ? 0.0f : M0, s1 = M1 == -INFINITY ? 0.0f : M1;
            const float a0 = exp2f(m0 - s0), b0 = exp2f(n0 - s0), a1 = exp2f(m1 - s1), b1 = exp2f(n1 - s1);
#pragma unroll
            for (int dn = 0; dn < DN; ++dn) {
                o[dn][0] = a0 * o[dn][0] + b0 * x[(dn * 4 + 0) * NT + tid];
                o[dn][1] = a0 * o[dn][1] + b0 * x[(dn * 4 + 1) * NT + tid];
                o[dn][2] = a1 * o[dn][2] + b1 * x[(dn * 4 + 2) * NT + tid];
                o[dn][3] = a1 * o[dn][3] + b1 * x[(dn * 4 + 3) * NT + tid];
            }
            l0 = a0 * l0 + b0 * k0;
            l1 = a1 * l1 + b1 * k1;
            m0 = M0;
            m1 = M1;
        }
    }
    if (csize == 1) {
        if (grp == 0) {
            const float i0 = 1.0f / l0, i1 = 1.0f / l1;
#pragma unroll
            for (int dn = 0; dn < DN; ++dn) {
                const int col = h * HD + dn * 8 + 2 * c4;
                if (r0 < nq)
                    *reinterpret_cast<__nv_bfloat162*>(out + (static_cast<size_t>(b) * T + q0 + r0) * qd + col) =
                        __floats2bfloat162_rn(o[dn][0] * i0, o[dn][1] * i0);
                if (r1 < nq)
                    *reinterpret_cast<__nv_bfloat162*>(out + (static_cast<size_t>(b) * T + q0 + r1) * qd + col) =
                        __floats2bfloat162_rn(o[dn][2] * i1, o[dn][3] * i1);
            }
        }
        if (sy.qkv_done && threadIdx.x == 0) pdl_wait();  // see AttnSync
        return;
    }
    // the CTA's partial into the first group's shared memory (its Q/K/V tiles are done)
    float* sO = reinterpret_cast<float*>(smem_attn);  // [AQ][HD]
    float* sML = sO + AQ * HD;                        // [AQ][2]
    if (grp == 0) {
#pragma unroll
        for (int dn = 0; dn < DN; ++dn) {
            const int col = dn * 8 + 2 * c4;
            *reinterpret_cast<float2*>(sO + r0 * HD + col) = make_float2(o[dn][0], o[dn][1]);
            *reinterpret_cast<float2*>(sO + r1 * HD + col) = make_float2(o[dn][2], o[dn][3]);
        }
        if (c4 == 0) {
            *reinterpret_cast<float2*>(sML + r0 * 2) = make_float2(m0, l0);
            *reinterpret_cast<float2*>(sML + r1 * 2) = make_float2(m1, l1);
        }
    }
    cluster_sync_all();  // every split's partial is in place
    if (tr) tr[kAtTicket] = global_ns();
    // This CTA merges output elements e = split * NTT + threadIdx.x (+ k * csize * NTT): row
    // e / V4, features 4 (e % V4) .. +3, over the csize partials in CTA order.  A row is one
    // aligned segment of V4 lanes; lane k of the segment reads partial k's (max, sum) and the
    // merge weights are shared by shuffles, so each partial's statistics cross the cluster once.
    constexpr int V4 = HD / 4;
    constexpr int NTT = PR * NT;
    const int ln = threadIdx.x & 31;
    const int seg0 = ln & ~(V4 - 1);
    uint32_t pb[kMaxCluster];
#pragma unroll
    for (int c = 0; c < kMaxCluster; ++c) pb[c] = c < csize ? dsmem_map(smem_u32(sO), c) : 0u;
    const int nel = nq * V4;
    // all lanes of a warp take the same passes (the shuffles); lanes past the end work on a
    // clamped row and store nothing
    for (int ew0 = split * NTT + (threadIdx.x & ~31); ew0 < nel; ew0 += csize * NTT) {
        const int e = ew0 + ln;
        const int r = min(e / V4, AQ - 1), i4 = e % V4;
        float mk = -INFINITY, lk = 0.0f;
        if (i4 < csize) {
            const float2 v = dsmem_ld2(dsmem_map(smem_u32(sML + r * 2), static_cast<uint32_t>(i4)));
            mk = v.x;
            lk = v.y;
        }
        float4 ov[kMaxCluster];
#pragma unroll
        for (int c = 0; c < kMaxCluster; ++c)
            if (c < csize) ov[c] = dsmem_ld4(pb[c] + static_cast<uint32_t>((r * HD + i4 * 4) * 4));
        float M = mk;  // over the first 8 lanes of the segment (csize <= 8)
        M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 1));
        M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 2));
        M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, 4));
        M = __shfl_sync(0xffffffffu, M, seg0);
        const float wk = mk == -INFINITY ? 0.0f : exp2f(mk - M);  // a share without keys: 0
        float L = wk * lk;
        L += __shfl_xor_sync(0xffffffffu, L, 1);
        L += __shfl_xor_sync(0xffffffffu, L, 2);
        L += __shfl_xor_sync(0xffffffffu, L, 4);
        L = __shfl_sync(0xffffffffu, L, seg0);
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int c = 0; c < kMaxCluster; ++c) {
            if (c < csize) {
                const float w = __shfl_sync(0xffffffffu, wk, seg0 + c);
                acc.x += w * ov[c].x;
                acc.y += w * ov[c].y;
                acc.z += w * ov[c].z;
                acc.w += w * ov[c].w;
            }
        }
        if (e < nel) {
            const float inv = 1.0f / L;
            __nv_bfloat16* op = out + (static_cast<size_t>(b) * T + q0 + r) * qd + h * HD + i4 * 4;
            *reinterpret_cast<__nv_bfloat162*>(op) = __floats2bfloat162_rn(acc.x * inv, acc.y * inv);
            *reinterpret_cast<__nv_bfloat162*>(op + 2) = __floats2bfloat162_rn(acc.z * inv, acc.w * inv);
        }
    }
    if (tr) tr[kAtMergeLoop] = global_ns();
    cluster_sync_all();  // no CTA leaves while its partials may still be read
    if (tr) tr[kAtMerged] = global_ns();
    if (sy.qkv_done && threadIdx.x == 0) pdl_wait();  // see AttnSync
}

static size_t attn_smem(int nw, int nb, int pr, int hd) {
    return static_cast<size_t>(pr) * (nw * 16 + 2 * nb * kAK) * hd * 2;
}

template <int HD, int NW, int NB, int PR>
static cudaError_t attn_attr() {
    return cudaFuncSetAttribute(reinterpret_cast<const void*>(k_attn<HD, NW, NB, PR>),
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(attn_smem(NW, NB, PR, HD)));
}

cudaError_t attn_init_attrs() {
    cudaError_t e = attn_tc_init_attrs();
    if (e == cudaSuccess) e = attn_attr<128, 2, 1, 1>();
    if (e == cudaSuccess) e = attn_attr<128, 2, 1, 2>();
    if (e == cudaSuccess) e = attn_attr<128, 2, 2, 1>();
    if (e == cudaSuccess) e = attn_attr<128, 4, 1, 1>();
    if (e == cudaSuccess) e = attn_attr<128, 4, 2, 1>();
    if (e == cudaSuccess) e = attn_attr<64, 2, 1, 1>();
    if (e == cudaSuccess) e = attn_attr<64, 2, 1, 2>();
    if (e == cudaSuccess) e = attn_attr<64, 2, 2, 1>();
    if (e == cudaSuccess) e = attn_attr<64, 4, 1, 1>();
    if (e == cudaSuccess) e = attn_attr<64, 4, 2, 1>();
    return e;
}

AttnPlan attn_plan(int B, int T, int H, int hd, int max_keys, int sms) {
    // long key ranges (head dim 128) go to the tensor-core kernel; on short ones, a few
    // sub-blocks per CTA, the mma.sync kernel has less latency per sub-block
    if (hd == 128 && max_keys >= kTcMinKeys) return attn_plan_tc(B, T, H, max_keys, sms);
    AttnPlan a{};
    // two warps (32 query rows) for the short windows of cached decoding, four otherwise: a
    // 64-token window is one query tile, so its keys and values are read once
    a.nw = T <= 32 ? 2 : 4;
    a.qtiles = (T + a.nw * 16 - 1) / (a.nw * 16);
    const int units = B * H * a.qtiles;
    const int blocks = (max_keys + kAK - 1) / kAK;
    a.pairs = 1;
    a.nb = 1;
    if (a.nw == 2 && blocks >= 2 && units * ((blocks + 1) / 2) <= sms + sms / 4 && (blocks + 1) / 2 <= kMaxCluster) {
        // few (sequence, head) units and a short prefix: one CTA per about two sub-blocks, its
        // two warp pairs taking one sub-block each (about one CTA per SM)
        a.pairs = 2;
        a.csize = (blocks + 1) / 2;
        return a;
    }
    // key splits (cluster size): about two CTAs per SM, at most one split per sub-block
    int c = (2 * sms) / units;
    if (c > kMaxCluster) c = kMaxCluster;
    if (c > blocks) c = blocks;
    if (c < 1) c = 1;
    a.csize = c;
    // long key ranges per CTA keep two sub-blocks of K and V in flight
    a.nb = (blocks + c - 1) / c >= 3 ? 2 : 1;
    return a;
}

template <int HD, int NW, int NB, int PR>
static cudaError_t attn_go(cudaLaunchConfig_t& cfg, const __nv_bfloat16* q, const __nv_bfloat16* kc,
                           const __nv_bfloat16* vc, const int* seq_kv, __nv_bfloat16* out, int T, int H, int Hkv,
                           int cap, const AttnPlan& a, unsigned long long* trace, const AttnSync& sy, int* status) {
    cfg.blockDim = dim3(PR * NW * 32);
    cfg.dynamicSmemBytes = attn_smem(NW, NB, PR, HD);
    return cudaLaunchKernelEx(&cfg, k_attn<HD, NW, NB, PR>, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a.qtiles, a.csize,
                              a.qx, trace, sy, status);
}

cudaError_t launch_attention(const __nv_bfloat16* q, const __nv_bfloat16* kc, const __nv_bfloat16* vc,
                             const int* seq_kv, __nv_bfloat16* out, int B, int T, int H, int Hkv, int hd, int cap,
                             const AttnPlan& a, cudaStream_t st, bool pdl, unsigned long long* trace, int* status,
                             const AttnSync* sync) {
    if (Hkv < 1 || H % Hkv) return cudaErrorInvalidValue;
    AttnSync sy{};
    if (sync && sync->qkv_done) {
        if (!sync->epoch || sync->qkv_ntile < 1 || sync->qkv_ntiles < 1) return cudaErrorInvalidValue;
        sy = *sync;
    }
    if (a.tc) {
        if (hd != 128) return cudaErrorInvalidValue;
        return launch_attention_tc(q, kc, vc, seq_kv, out, B, T, H, Hkv, cap, a, st, pdl, trace, status);
    }
    if (a.csize < 1 || a.csize > kMaxCluster || (a.nw != 2 && a.nw != 4) || (a.nb != 1 && a.nb != 2) ||
        (a.pairs != 1 && a.pairs != 2) || (a.pairs == 2 && (a.nw != 2 || a.nb != 1)) || (hd != 64 && hd != 128))
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
    if (a.pairs == 2)
        return hd == 128 ? attn_go<128, 2, 1, 2>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status)
                         : attn_go<64, 2, 1, 2>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status);
    const int key = (hd == 128 ? 4 : 0) + (a.nw == 4 ? 2 : 0) + (a.nb == 2 ? 1 : 0);
    switch (key) {
        case 0: return attn_go<64, 2, 1, 1>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status);
        case 1: return attn_go<64, 2, 2, 1>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status);
        case 2: return attn_go<64, 4, 1, 1>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status);
        case 3: return attn_go<64, 4, 2, 1>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status);
        case 4: return attn_go<128, 2, 1, 1>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status);
        case 5: return attn_go<128, 2, 2, 1>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status);
        case 6: return attn_go<128, 4, 1, 1>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status);
        default: return attn_go<128, 4, 2, 1>(cfg, q, kc, vc, seq_kv, out, T, H, Hkv, cap, a, trace, sy, status);
    }
}

// ------------------------------------------------------------------ LM head
// Merge the per-tile (max, sum exp, argmax) of each token over the vocab
// tiles in a fixed tree: argmax excludes the mask id, ties go to the lowest
// id; conf = 1 / sum; tokconf = exp(z_cur - max) / sum.
__device__ __forceinline__ void lse_merge(float& m, float& s, int& i, float m2, float s2, int i2) {
    if (m2 == -INFINITY) return;
    if (m == -INFINITY) {
        m = m2; s = s2; i = i2;
        return;
    }
    if (m2 > m) {
        s = s * expf(m - m2) + s2;
        m = m2;
        i = i2;
    } else if (m2 == m) {
        s += s2;
        i = min(i, i2);
    } else {
        s += s2 * expf(m2 - m);
    }
}

__global__ void __launch_bounds__(256) k_lmhead_reduce(const float* __restrict__ part, const float* __restrict__ zcur,
                                                        const int* __restrict__ cur_tok, int m_tiles, int mask_id,
                                                        int* x0, float* conf, float* tokconf, const int* row_map,
                                                        const int* n_rows) {
    pdl_wait();
    pdl_launch_dependents();
    __shared__ float sm_m[8], sm_s[8];
    __shared__ int sm_i[8];
    const int col = blockIdx.x;  // the head's token column (a compacted row with a row map)
    if (row_map && col >= *n_rows) return;
    const int out = row_map ? row_map[col] : col;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float m = -INFINITY, s = 0.0f;
    int idx = INT_MAX;
    const float* pc = part + static_cast<size_t>(col) * m_tiles * 3;
    for (int t = threadIdx.x; t < m_tiles; t += blockDim.x)
        lse_merge(m, s, idx, pc[t * 3], pc[t * 3 + 1], __float_as_int(pc[t * 3 + 2]));
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const float m2 = __shfl_down_sync(0xffffffffu, m, off);
        const float s2 = __shfl_down_sync(0xffffffffu, s, off);
        const int i2 = __shfl_down_sync(0xffffffffu, idx, off);
        if ((lane & (2 * off - 1)) == 0 && lane + off < 32) lse_merge(m, s, idx, m2, s2, i2);
    }
    if (lane == 0) {
        sm_m[warp] = m;
        sm_s[warp] = s;
        sm_i[warp] = idx;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        m = sm_m[0];
        s = sm_s[0];
        idx = sm_i[0];
        for (int w = 1; w < static_cast<int>(blockDim.x >> 5); ++w) lse_merge(m, s, idx, sm_m[w], sm_s[w], sm_i[w]);
        x0[out] = idx;
        conf[out] = 1.0f / s;
        const int cur = cur_tok[col];
        tokconf[out] = (cur >= 0 && cur != mask_id) ? expf(zcur[col] - m) / s : 0.0f;
    }
}

cudaError_t launch_lmhead_reduce(const float* lm_part, const float* zcur, const int* cur_tok, int m_tiles, int N,
                                 int mask_id, int* x0, float* conf, float* tokconf, cudaStream_t st, bool pdl,
                                 const int* row_map, const int* n_rows) {
    return launch_k(k_lmhead_reduce, dim3(N), dim3(256), 0, st, pdl, lm_part, zcur, cur_tok, m_tiles, mask_id, x0, conf,
                    tokconf, row_map, n_rows);
}

// ------------------------------------------------------------------ selective logits skipping
// One CTA lists the rows (b T + t) that need a decision, in ascending order: window row t < Tw
// is needed when its position's state is MASKED (1), COMMITTED (2) or DRAFT (4); rows t >= Tw
// (tracked refresh rows) always.  Skipped rows get x0 = -1, conf = tokconf = 0.
__global__ void __launch_bounds__(1024) k_sls_map(const uint8_t* st, int ld, const int* seq_kv, int use_cache, int B,
                                                  int Tw, int T, int* row_map, int* n_rows, int* x0, float* conf,
                                                  float* tokconf) {
    pdl_wait();
    pdl_launch_dependents();
    __shared__ int s_warp[32];
    __shared__ int s_base;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    if (threadIdx.x == 0) s_base = 0;
    __syncthreads();
    const int N = B * T;
    for (int base = 0; base < N; base += blockDim.x) {
        const int row = base + static_cast<int>(threadIdx.x);
        bool need = false;
        if (row < N) {
            const int b = row / T, t = row - b * T;
            if (t >= Tw) {
                need = true;
            } else {
                const int w0 = use_cache ? seq_kv[b] : 0;
                const uint8_t s = st[static_cast<size_t>(b) * ld + w0 + t];
                need = s == 1 || s == 2 || s == 4;
            }
        }
        const uint32_t bal = __ballot_sync(0xffffffffu, need);
        if (lane == 0) s_warp[warp] = __popc(bal);
        __syncthreads();
        int before = s_base, tot = 0;
        for (int w = 0; w < nw; ++w) {
            const int c = s_warp[w];
            if (w < warp) before += c;
            tot += c;
        }
        before += __popc(bal & ((1u << lane) - 1u));
        if (need) {
            row_map[before] = row;
        } else if (row < N) {
            x0[row] = -1;
            conf[row] = 0.0f;
            tokconf[row] = 0.0f;
        }
        __syncthreads();  // every thread has read s_base and s_warp
        if (threadIdx.x == 0) s_base += tot;
        __syncthreads();
    }
    if (threadIdx.x == 0) *n_rows = s_base;
}

cudaError_t launch_sls_map(const uint8_t* st, int ld, const int* seq_kv, int use_cache, int B, int Tw, int T,
                           int* row_map, int* n_rows, int* x0, float* conf, float* tokconf, cudaStream_t stream) {
    return launch_k(k_sls_map, dim3(1), dim3(1024), 0, stream, true, st, ld, seq_kv, use_cache, B, Tw, T, row_map,
                    n_rows, x0, conf, tokconf);
}

// One warp per compact row j < pad_to: rows j < n copy activation row row_map[j] (d bf16, 16-byte
// pieces), its n_sq RMSNorm statistics (stride N) and current id; rows n <= j < pad_to become
// zero activations with unit statistics and id -1 (finite, and never reduced).
__global__ void __launch_bounds__(256) k_sls_gather(const int* row_map, const int* n_rows, int N, int pad_to, int d,
                                                    const __nv_bfloat16* xn, const float* sq, int n_sq,
                                                    const int* cur, __nv_bfloat16* xc, float* sqc, int* curc) {
    pdl_wait();
    pdl_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int j = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int n = *n_rows;
    const int pad_end = (n + pad_to - 1) / pad_to * pad_to;  // the end of the last token tile in use
    if (j >= pad_end || j >= N) return;
    const int n16 = d / 8;
    uint4* dst = reinterpret_cast<uint4*>(xc + static_cast<size_t>(j) * d);
    if (j < n) {
        const int row = row_map[j];
        const uint4* src = reinterpret_cast<const uint4*>(xn + static_cast<size_t>(row) * d);
        for (int i = lane; i < n16; i += 32) dst[i] = src[i];
        for (int t = lane; t < n_sq; t += 32) sqc[static_cast<size_t>(t) * N + j] = sq[static_cast<size_t>(t) * N + row];
        if (lane == 0) curc[j] = cur[row];
    } else {
        for (int i = lane; i < n16; i += 32) dst[i] = make_uint4(0u, 0u, 0u, 0u);
        for (int t = lane; t < n_sq; t += 32) sqc[static_cast<size_t>(t) * N + j] = 1.0f;
        if (lane == 0) curc[j] = -1;
    }
}

cudaError_t launch_sls_gather(const int* row_map, const int* n_rows, int N, int pad_to, int d,
                              const __nv_bfloat16* xn, const float* sq, int n_sq, const int* cur,
                              __nv_bfloat16* xc, float* sqc, int* curc, cudaStream_t stream) {
    if (N < 1 || pad_to < 1 || d % 8) return cudaErrorInvalidValue;
    return launch_k(k_sls_gather, dim3((N + 7) / 8), dim3(256), 0, stream, true, row_map, n_rows, N, pad_to, d, xn,
                    sq, n_sq, cur, xc, sqc, curc);
}

// ------------------------------------------------------------------ commit pass
// One CTA per sequence.  Order (all on this step's decisions):
//  1. revision (theta_remask > 0, not the last step): COMMITTED tokens of the
//     current block with tokconf >= theta_stable become STABLE; of those below
//     theta_remask, the remask_max lowest (ties: lower position) are re-masked;
//  2. schedule mode: k = ceil(m / (S - step)) for the m masked positions of
//     the block, and the k masked positions with the highest conf (ties: lower
//     position) take their argmax and become COMMITTED;
//  3. threshold mode (staged token stabilization): the masked positions with
//     conf >= theta_visible take their argmax and become COMMITTED (STABLE at
//     conf >= theta_stable); when there is none, the single most confident one
//     (ties: lower position) becomes COMMITTED;
//  4. with the prefix cache and lookahead on, each future block inside the
//     window drafts its single most confident masked position.
__global__ void __launch_bounds__(256) k_commit(CommitArgs a) {
    pdl_wait();
    pdl_launch_dependents();
    const int b = blockIdx.x;
    int* tok = a.tok + static_cast<size_t>(b) * a.ld;
    uint8_t* st = a.st + static_cast<size_t>(b) * a.ld;
    int* plan = a.plan + b * 4;
    const int c0 = plan[0], c1 = plan[1], step = plan[2];
    const int n = c1 - c0;  // <= kMaxBlock (checked by the host)
    const int w0 = a.use_cache ? a.seq_kv[b] : 0;
    const int* x0 = a.x0 + static_cast<size_t>(b) * a.Tq;
    const float* conf = a.conf + static_cast<size_t>(b) * a.Tq;
    const float* tc = a.tokconf + static_cast<size_t>(b) * a.Tq;
    __shared__ int s_cnt[8];
    __shared__ uint8_t s_sel[kMaxBlock];
    __shared__ uint8_t s_vis[kMaxBlock];  // continuous sliding: block positions visible at the forward
    if (threadIdx.x < 8) s_cnt[threadIdx.x] = 0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const int p = c0 + i;
        s_vis[i] = p >= w0 && (st[p] == 2 || st[p] == 3);
    }
    __syncthreads();
    // the revision reaches only the block positions inside the window (sliding moves w0 past c0)
    if (a.theta_remask > 0.0f && step < a.S - 1) {
        for (int i = threadIdx.x; i < n; i += blockDim.x) {
            const int p = c0 + i;
            if (p >= w0 && st[p] == 2 && tc[p - w0] >= a.theta_stable) {
                st[p] = 3;
                atomicAdd(&s_cnt[2], 1);
            }
        }
        __syncthreads();
        // candidates ranked by (tokconf ascending, position ascending)
        for (int i = threadIdx.x; i < n; i += blockDim.x) {
            const int p = c0 + i;
            uint8_t sel = 0;
            if (p >= w0 && st[p] == 2 && tc[p - w0] < a.theta_remask) {
                const float vp = tc[p - w0];
                int rank = 0;
                for (int qq = max(c0, w0); qq < c1; ++qq) {
                    if (qq == p || st[qq] != 2) continue;
                    const float vq = tc[qq - w0];
                    if (!(vq < a.theta_remask)) continue;
                    if (vq < vp || (vq == vp && qq < p)) ++rank;
                }
                sel = rank < a.remask_max;
            }
            s_sel[i] = sel;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < n; i += blockDim.x) {
            if (s_sel[i]) {
                st[c0 + i] = 1;
                tok[c0 + i] = a.mask_id;
                atomicAdd(&s_cnt[1], 1);
            }
        }
        __syncthreads();
    }
    int mloc = 0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) mloc += st[c0 + i] == 1;
    atomicAdd(&s_cnt[5], mloc);
    __syncthreads();
    const int m = s_cnt[5];
    if (a.commit_mode == 1) {
        for (int i = threadIdx.x; i < n; i += blockDim.x) {
            const int p = c0 + i;
            const float v = conf[p - w0];
            if (st[p] == 1 && v >= a.theta_visible) {
                tok[p] = x0[p - w0];
                const bool stable = v >= a.theta_stable;
                st[p] = stable ? 3 : 2;
                atomicAdd(&s_cnt[0], 1);
                if (stable) atomicAdd(&s_cnt[2], 1);
            }
        }
        __syncthreads();
        if (s_cnt[0] == 0 && m > 0 && threadIdx.x < 32) {  // the most confident masked position
            float bv = -INFINITY;
            int bp = INT_MAX;
            for (int p = c0 + static_cast<int>(threadIdx.x); p < c1; p += 32) {
                if (st[p] != 1) continue;
                const float v = conf[p - w0];
                if (v > bv || (v == bv && p < bp)) {
                    bv = v;
                    bp = p;
                }
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
                const int op = __shfl_xor_sync(0xffffffffu, bp, off);
                if (ov > bv || (ov == bv && op < bp)) {
                    bv = ov;
                    bp = op;
                }
            }
            if (threadIdx.x == 0 && bp != INT_MAX) {
                tok[bp] = x0[bp - w0];
                st[bp] = 2;
                s_cnt[0] = 1;
            }
        }
        __syncthreads();
    }
    const int left = a.S - step;
    const int k = a.commit_mode == 1 || m == 0 ? 0 : (left <= 1 ? m : (m + left - 1) / left);
    // schedule mode: the k masked positions ranked by (conf descending, position ascending)
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const int p = c0 + i;
        uint8_t sel = 0;
        if (st[p] == 1) {
            const float vp = conf[p - w0];
            int rank = 0;
            for (int qq = c0; qq < c1; ++qq) {
                if (qq == p || st[qq] != 1) continue;
                const float vq = conf[qq - w0];
                if (vq > vp || (vq == vp && qq < p)) ++rank;
            }
            sel = rank < k;
        }
        s_sel[i] = sel;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        if (s_sel[i]) {
            const int p = c0 + i;
            tok[p] = x0[p - w0];
            st[p] = 2;
            atomicAdd(&s_cnt[0], 1);
        }
    }
    __syncthreads();
    // drafts for the future blocks inside the window
    if (a.use_cache && (a.spec_blocks > 0 || a.slide_kv) && threadIdx.x < 32) {
        const int w1 = w0 + a.T;
        for (int d0 = c1; d0 < w1; d0 += a.block_len) {
            const int d1 = min(d0 + a.block_len, w1);
            float bv = -INFINITY;
            int bp = INT_MAX;
            for (int p = d0 + static_cast<int>(threadIdx.x); p < d1; p += 32) {
                if (st[p] != 1) continue;
                const float v = conf[p - w0];
                if (v > bv || (v == bv && p < bp)) {
                    bv = v;
                    bp = p;
                }
            }
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) {
                const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
                const int op = __shfl_xor_sync(0xffffffffu, bp, off);
                if (ov > bv || (ov == bv && op < bp)) {
                    bv = ov;
                    bp = op;
                }
            }
            if (threadIdx.x == 0 && bp != INT_MAX) {
                tok[bp] = x0[bp - w0];
                st[bp] = 4;
                s_cnt[3] += 1;
            }
            __syncwarp();
        }
    }
    __syncthreads();
    // sparse cache refresh: the tracked prefix positions, rows Tw + r, re-scored; those that
    // keep their id have their refreshed K/V merged after this kernel
    for (int r = threadIdx.x; r < a.R; r += blockDim.x) {
        const int p = a.trk[b * a.R + r];
        int merge = 0;
        if (p >= 0) {
            const float v = tc[a.T + r];
            const int x = x0[a.T + r];
            merge = 1;
            if (v >= a.theta_stable) {
                st[p] = 3;
                atomicAdd(&s_cnt[2], 1);
            } else if (a.theta_remask > 0.0f && v < a.theta_remask && x != tok[p]) {
                tok[p] = x;
                merge = 0;
                atomicAdd(&s_cnt[7], 1);
            }
            if (merge) atomicAdd(&s_cnt[6], 1);
        }
        a.merge[b * a.R + r] = merge;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int* o = a.outs + b * 8;
        o[0] = s_cnt[0];
        o[1] = s_cnt[1];
        o[2] = s_cnt[2];
        o[3] = s_cnt[3];
        o[5] = m - s_cnt[0];
        o[4] = o[5] == 0;
        o[6] = s_cnt[6];
        o[7] = s_cnt[7];
        plan[2] = step + 1;
        if (a.slide_kv && w0 >= c0) {
            // continuous sliding: the leading run of block positions visible at the forward and
            // still visible joins the cache (its K/V were written there by this step's forward)
            int adv = 0;
            while (w0 + adv < c1 && s_vis[w0 + adv - c0] && (st[w0 + adv] == 2 || st[w0 + adv] == 3)) ++adv;
            a.slide_kv[b] = w0 + adv;
        }
    }
}

// ------------------------------------------------------------------ sparse cache refresh
// One CTA per sequence b: trk[b R + r] = the r-th position p < seq_kv[b] whose state is
// COMMITTED (ascending), -1 past the last.  Positions are scanned 256 at a time with a
// block-wide prefix count.
__global__ void __launch_bounds__(256) k_scr_select(const uint8_t* st_all, int ld, const int* seq_kv, int* trk_all,
                                                    int R) {
    pdl_wait();
    pdl_launch_dependents();
    __shared__ int s_warp[8];
    __shared__ int s_base;
    const int b = blockIdx.x;
    const uint8_t* st = st_all + static_cast<size_t>(b) * ld;
    int* trk = trk_all + b * R;
    const int kv = seq_kv[b];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) s_base = 0;
    for (int r = threadIdx.x; r < R; r += blockDim.x) trk[r] = -1;
    __syncthreads();
    for (int p0 = 0; p0 < kv; p0 += blockDim.x) {
        const int p = p0 + static_cast<int>(threadIdx.x);
        const bool hit = p < kv && st[p] == 2;
        const unsigned bal = __ballot_sync(0xffffffffu, hit);
        if (lane == 0) s_warp[warp] = __popc(bal);
        __syncthreads();
        int before = s_base;
        for (int w = 0; w < warp; ++w) before += s_warp[w];
        const int idx = before + __popc(bal & ((1u << lane) - 1u));
        if (hit && idx < R) trk[idx] = p;
        __syncthreads();
        if (threadIdx.x == 0) {
            int tot = 0;
            for (int w = 0; w < 8; ++w) tot += s_warp[w];
            s_base += tot;
        }
        __syncthreads();
        if (s_base >= R) break;
    }
}

cudaError_t launch_scr_select(const uint8_t* st, int ld, const int* seq_kv, int* trk, int B, int R,
                              cudaStream_t stream) {
    return launch_k(k_scr_select, dim3(B), dim3(256), 0, stream, true, st, ld, seq_kv, trk, R);
}

// Grid (R, L, B): row r of sequence b in layer l, when merged, copies its K and V rows of every
// head (hd elements each) from the side buffers into the cache at position trk[b R + r].
__global__ void __launch_bounds__(128) k_scr_merge(const __nv_bfloat16* side, __nv_bfloat16* cache, const int* trk,
                                                   const int* merge, int B, int kv_B, int H, int hd, int cap, int R) {
    pdl_wait();
    pdl_launch_dependents();
    const int r = blockIdx.x, l = blockIdx.y, b = blockIdx.z;
    const int p = trk[b * R + r];
    if (p < 0 || !merge[b * R + r]) return;
    const size_t side_layer = static_cast<size_t>(2) * B * H * R * hd;
    const size_t cache_half = static_cast<size_t>(kv_B) * H * cap * hd;
    const int n4 = hd / 8;  // 16-byte pieces per head row
    for (int e = threadIdx.x; e < 2 * H * n4; e += blockDim.x) {
        const int which = e / (H * n4), rem = e - which * H * n4;
        const int h = rem / n4, i = rem - h * n4;
        const uint4* src = reinterpret_cast<const uint4*>(
                               side + l * side_layer + ((static_cast<size_t>(which) * B + b) * H + h) * R * hd +
                               static_cast<size_t>(r) * hd) + i;
        uint4* dst = reinterpret_cast<uint4*>(cache + (static_cast<size_t>(2 * l + which)) * cache_half +
                                              ((static_cast<size_t>(b) * H + h) * cap + p) * hd) + i;
        *dst = *src;
    }
}

cudaError_t launch_scr_merge(const __nv_bfloat16* side, __nv_bfloat16* cache, const int* trk, const int* merge, int L,
                             int B, int kv_B, int H, int hd, int cap, int R, cudaStream_t stream) {
    if (R < 1 || hd % 8 || B < 1 || B > kv_B) return cudaErrorInvalidValue;
    return launch_k(k_scr_merge, dim3(R, L, B), dim3(128), 0, stream, true, side, cache, trk, merge, B, kv_B, H, hd,
                    cap, R);
}

cudaError_t launch_commit(const CommitArgs& a, cudaStream_t st, bool pdl) {
    return launch_k(k_commit, dim3(a.B), dim3(256), 0, st, pdl, a);
}

}  // namespace dllm

namespace dllm {

// Start a block on every sequence: plan = {c0, c1, step 0}; drafts inside the
// block become COMMITTED; snapshot the window region for rewinds.
__global__ void k_begin_block(int* tok, uint8_t* st, int* snap_tok, uint8_t* snap_st, int ld, int n_pos, int* plan,
                              int c0, int c1) {
    pdl_wait();
    pdl_launch_dependents();
    const int b = blockIdx.x;
    int* t = tok + static_cast<size_t>(b) * ld;
    uint8_t* s = st + static_cast<size_t>(b) * ld;
    for (int p = c0 + threadIdx.x; p < c1; p += blockDim.x)
        if (s[p] == 4) s[p] = 2;
    __syncthreads();
    for (int p = threadIdx.x; p < n_pos; p += blockDim.x) {
        snap_tok[static_cast<size_t>(b) * ld + p] = t[p];
        snap_st[static_cast<size_t>(b) * ld + p] = s[p];
    }
    if (threadIdx.x == 0) {
        plan[b * 4 + 0] = c0;
        plan[b * 4 + 1] = c1;
        plan[b * 4 + 2] = 0;
    }
}

cudaError_t launch_begin_block(int* tok, uint8_t* st, int* snap_tok, uint8_t* snap_st, int ld, int n_pos, int* plan,
                               int B, int c0, int c1, cudaStream_t stream) {
    return launch_k(k_begin_block, dim3(B), dim3(256), 0, stream, true, tok, st, snap_tok, snap_st, ld, n_pos, plan, c0, c1);
}

__global__ void k_rewind(int* tok, uint8_t* st, const int* snap_tok, const uint8_t* snap_st, int ld, int n_pos,
                         int* plan) {
    pdl_wait();
    pdl_launch_dependents();
    const int b = blockIdx.x;
    for (int p = threadIdx.x; p < n_pos; p += blockDim.x) {
        tok[static_cast<size_t>(b) * ld + p] = snap_tok[static_cast<size_t>(b) * ld + p];
        st[static_cast<size_t>(b) * ld + p] = snap_st[static_cast<size_t>(b) * ld + p];
    }
    if (threadIdx.x == 0) plan[b * 4 + 2] = 0;
}

cudaError_t launch_rewind(int* tok, uint8_t* st, const int* snap_tok, const uint8_t* snap_st, int ld, int n_pos,
                          int* plan, int B, cudaStream_t stream) {
    return launch_k(k_rewind, dim3(B), dim3(256), 0, stream, true, tok, st, snap_tok, snap_st, ld, n_pos, plan);
}

__global__ void k_set_kv_len(int* seq_kv, int B, int v) {
    pdl_wait();
    pdl_launch_dependents();
    int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b < B) seq_kv[b] = v;
}

cudaError_t launch_set_kv_len(int* seq_kv, int B, int v, cudaStream_t stream) {
    return launch_k(k_set_kv_len, dim3((B + 127) / 128), dim3(128), 0, stream, true, seq_kv, B, v);
}

}  // namespace dllm
