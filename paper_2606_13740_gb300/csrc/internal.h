// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <utility>

namespace dllm {

constexpr int kMaxBlock = 4096;
constexpr int kStatusTimeout = 1;  // device status word bits
constexpr int kStatusBadIndex = 2;  // longest current block the commit pass handles

// ---------------------------------------------------------------- weight storage
// The context's projection weights are stored tile-major: the 128-row x 64-column tile
// (m-tile r/128, k-block c/64) of a [rows][K] matrix is 16 KB at ((r/128)*kb + c/64)*8192
// elements (kb = ceil(K/64), columns past K zero), row r%128 of the tile 64 elements long,
// and the 16-byte chunk (c%64)/8 of that row placed at chunk ((c%64)/8) ^ (r%8).  That is the
// 128-byte-swizzled K-major image the UMMA shared-memory descriptor reads, so a tile moves
// from HBM to shared memory as one contiguous copy (long DRAM bursts instead of 128 rows of
// 128 bytes).
__host__ __device__ inline size_t tiled_index(int r, int c, int kb) {
    return (static_cast<size_t>(r >> 7) * kb + (c >> 6)) * 8192 + static_cast<size_t>(r & 127) * 64 +
           ((((c & 63) >> 3) ^ (r & 7)) << 3) + (c & 7);
}

// ---------------------------------------------------------------- 4-bit weight storage
// A 128-row x 64-column tile of 4-bit block-quantised weights (32 weights of a row share one
// bf16 scale d; a weight is a 4-bit code q standing for d * (q - 8)) is kQ4TileBytes: first the
// codes, 32-bit word (c16, r) = the 8 codes of row r, columns 8 c16 .. 8 c16 + 7, at word
// c16 * 128 + r, column 8 c16 + j in bits 4 (j / 2) + 16 (j % 2) .. +3 (so that one mask and
// one OR turn a shifted word into the bf16 pair 128 + q of two neighbouring columns); then the
// scales, bf16 (b, r) for columns 32 b .. 32 b + 31 of row r at 4096 + 2 (b * 128 + r).
// Tiles are stored tile-major as for bf16 ((m-tile * kb + k-block) * kQ4TileBytes).
constexpr int kQ4TileBytes = 4096 + 512;
__host__ __device__ inline int q4_code_shift(int j) { return 4 * (j >> 1) + 16 * (j & 1); }

// ---------------------------------------------------------------- GEMM
// D = W * X^T on tensor cores: W bf16 [M][K] (weights, rows padded to 128),
// X bf16 [N][K] (tokens).  Row m of D is an output feature, column n a token.
enum EpiKind { EPI_F32 = 0, EPI_RESID = 1, EPI_QKV = 2, EPI_SWIGLU = 3, EPI_LMHEAD = 4 };

struct EpiArgs {
    float* out;          // EPI_F32: D[n][m] (ld = ld_out); EPI_RESID: residual x[n][m] += D
    int ld_out;
    // EPI_RESID also writes xb = bf16(x) [n][m] (the next projection's operand) and
    // sq_out[m_tile][n] = sum over the tile's 128 rows of x^2 (RMSNorm statistics)
    __nv_bfloat16* xb;
    float* sq_out;
    // QKV / SWIGLU / LMHEAD: per-token RMSNorm scale rsqrt(sum_t sq_in[t][n] / norm_dim + eps)
    // applied to the accumulators (the operand is bf16 of the un-normalised x); null = none
    const float* sq_in;
    int n_sq, norm_dim;
    float eps;
    // EPI_QKV: rows [0,qd) q, [qd,qd+kvd) k, [qd+kvd,qd+2kvd) v (qd = H*hd, kvd = Hkv*hd: under
    // grouped-query attention fewer K/V heads than query heads); rotate-half RoPE on q, k.
    // Inside each head the rows are interleaved: row 2j is feature j, row 2j+1 feature j + hd/2
    __nv_bfloat16* q;    // [B][H][T][hd]
    __nv_bfloat16* kc;   // layer's K cache base: [B][Hkv][cap][hd]
    __nv_bfloat16* vc;
    const int* seq_kv;   // per-sequence first window position (kv_len)
    int T, H, hd, cap;
    int Hkv;             // K/V heads (a multiple of 128 / hd rows each part: Hkv * hd % 128 == 0)
    int v_row0;          // first v row: qd + Hkv * hd
    int n_seq;           // sequences (B), <= 256
    const float* theta;  // [hd/2]: rotation of feature pair j at position p is p * theta[j]
    // EPI_SWIGLU: tile k row 2f is gate feature 64k+f, row 2f+1 the matching up row
    __nv_bfloat16* h;    // [N][F]
    int F;
    // EPI_QKV with sparse cache refresh: of a sequence's T rows the first Tw are the window,
    // row Tw + r of sequence b is the prefix position trk[b R + r] (< 0: an unused row, no K/V
    // written), whose K and V go to kside / vside [B][Hkv][R][hd] instead of the cache
    int Tw, R;
    const int* trk;
    __nv_bfloat16* kside;
    __nv_bfloat16* vside;
    // EPI_LMHEAD
    float* lm_part;      // [N][m_tiles][3]: max, sum exp(z - max), argmax (as float bits)
    float* zcur;         // [N]: logit of the current token id
    const int* cur_tok;  // [N]
    float* logits;       // [N][V] or null
    int V, mask_id;
    // timeline trace (null = off): per CTA 16 %globaltimer stamps / ids, see kTr* in gemm_tc.cu
    unsigned long long* trace;
};

struct GemmPlan {
    int M, N, K;
    int ntile;           // token tile (UMMA N), multiple of 16, <= 256
    int m_tiles, n_tiles, kb;
    long long total;     // m_tiles * n_tiles * kb iterations of 64-wide K blocks
    int grid;            // CTAs (stream-K partition of the iterations)
    bool pdl;            // launch with programmatic dependent launch (the step's chain)
};

struct Scratch {
    float* partials;     // [grid][ntile*128]: one split partial per CTA (gemm_partial_floats)
    int* counters;       // tile tickets, one per 128-byte line ([m_tiles*n_tiles][32]), zero between launches
    size_t partial_floats;
    int counter_len;
};

// ---------------------------------------------------------------- chained projections
// One persistent launch (one CTA per SM) runs up to kMaxPhases projections back to back,
// e.g. output projection -> gate/up -> down -> the next layer's QKV.  The weight ring
// streams on from one phase into the next while the previous phase's split tiles are
// reduced and its epilogues run; the operand (X) of phase i, k-block k, is loaded once the
// tile of phase i-1 that produces it has published its completion flag.
constexpr int kMaxPhases = 4;
struct ChainPhase {
    GemmPlan p;          // from gemm_plan (grid <= the chain's grid)
    EpiArgs ep;
    int epi;             // EpiKind
    int dep_rows;        // X k-block k comes from tile (64k)/dep_rows of the previous phase (a power of two); 0: ready at launch
    int* done;           // [m_tiles][n_tiles] completion flags (value: the launch's tag); may be null
    // residual phases: done = the bf16 operand is written, done2 = also the fp32 residual and
    // the RMSNorm sums (what the later phases' epilogues read); null: done covers both
    int* done2;
    float* partials;     // [grid][ntile*128] split partials (a CTA contributes to at most one tile per phase)
    int* tickets;        // [m_tiles*n_tiles][32], zero between launches
    // non-null: the weights are stored tile-major (tiled_index) and each 16 KB tile arrives with
    // one contiguous bulk copy; null: row-major [M][K] through the chain's tensor map.  In a
    // 4-bit chain (ChainArgs::q4) the tiles are kQ4TileBytes each, laid out as described at
    // kQ4TileBytes.
    const void* w_tiles;
};
struct ChainArgs {
    int n_phases;
    int grid, stages, ntile, acc_cols, tmem_cols;
    int red_bytes;       // shared staging for split partials
    int x_cols;          // TMEM columns for the staged old residual (0: none)
    int stg_bytes;       // the epilogue's own output staging (0: it shares the partial staging)
    size_t smem;
    const int* epoch;    // device step counter; tag = *epoch * tag_mul + tag_add (null: tag = tag_add)
    int tag_mul, tag_add;
    int* status;
    // Rows resolved on the device (null: every phase's plan as given).  With it, the launch
    // reads the token count from here once its predecessor has finished, and every phase
    // covers only the token tiles that hold those rows (the rest of the iteration space is
    // re-split over the CTAs).  Used by the LM head over compacted rows.
    const int* dyn_rows;
    // Test hook for the bounded waits (null: off): the operand producer waits for *gate == the
    // launch's tag before its first load.  Given a word nobody writes, that wait runs out after
    // kWaitLimitCycles and the launch unwinds with kStatusTimeout, as any stalled wait would.
    const int* gate;
    // 4-bit weights (the block format of Q4_0, see kQ4TileBytes): the weight producer streams
    // raw 4.5 KB tiles into raw_stages slots, four more warps expand each into the bf16 A stage
    // the tensor cores read, and the operand tiles go through a ring of b_stages of their own
    int q4, raw_stages, b_stages;  // b_stages: the operand ring of the 4-bit kernel
    // 4-bit kernel: the expanded A stages in tensor memory from column a_col0 instead of shared
    // memory, where TMEM has the room; a stage there holds two consecutive k-blocks of a tile
    // (64 columns, the MMA reading A from there; raw slots of two tiles, raw_stages ==
    // stages, and operand stages of two k-blocks)
    int a_tmem, a_col0;
    ChainPhase ph[kMaxPhases];
};
struct ChainMaps {
    CUtensorMap w[kMaxPhases];
    CUtensorMap x[kMaxPhases];
};
// Fills grid, stages, ntile, acc_cols, x_cols, stg_bytes, tmem_cols, red_bytes and
// smem from the phases' plans for a shared-memory budget (bytes, <= 227 KB).  False if the
// phases do not share one token tiling.
bool chain_plan(ChainArgs& ca, int smem_budget);
constexpr int kChainSmemFull = 227 * 1024;    // one CTA per SM, deepest ring
constexpr int kChainSmemShared = 146 * 1024;  // leaves room for two attention CTAs beside it
cudaError_t chain_launch(const ChainMaps& maps, const ChainArgs& ca, cudaStream_t st, bool pdl);
cudaError_t chain_init_attrs();

// Tiling of one projection: token tiles of at most 256 (multiples of 32), 128 weight rows
// per tile, 64-wide k-blocks, grid = min(iterations, grid_max).
GemmPlan gemm_plan(int M, int N, int K, int grid_max, int epi);
// Split-partial floats a single-projection launch of plan p needs (a CTA contributes to at most
// one split tile, so one ntile x 128 slot per CTA); gemm_launch rejects a smaller Scratch.
inline size_t gemm_partial_floats(const GemmPlan& p) {
    return static_cast<size_t>(p.grid) * static_cast<size_t>(p.ntile) * 128;
}
bool make_tmap_bf16(CUtensorMap* tm, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows);
cudaError_t gemm_launch(int epi, const GemmPlan& p, const CUtensorMap& tmW, const CUtensorMap& tmX,
                        const EpiArgs& ep, const Scratch& scr, int* status, cudaStream_t st,
                        const int* gate = nullptr);

// ---------------------------------------------------------------- launches
// Every kernel is launched with programmatic stream serialisation (PDL): it may start
// while its predecessor drains, and waits (griddepcontrol.wait) before touching data the
// predecessor writes.  set_pdl(false) launches them plainly.
void set_pdl(bool on);
// Single projections (dllm_op_gemm_*): true = the chain's 146 KB plan, false = 227 KB.
void set_stream_smem(bool coresident);
bool pdl_enabled();

template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*k)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, bool pdl,
                            Args&&... args) {
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = (pdl && pdl_enabled()) ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k, std::forward<Args>(args)...);
}

// ---------------------------------------------------------------- other kernels
// Seeded weights (rows_phys x cols, see k_init_weight for the row orders), stored tile-major
// (tiled_index; rows_phys a multiple of 128) when `tiled`, else row-major.
cudaError_t launch_init_weight(__nv_bfloat16* dst, int mode, int rows_phys, int cols, int logical_rows,
                               uint64_t seed, uint64_t tid0, int qd, int kvd, int hd, bool tiled, cudaStream_t st);
// The same weights in the 4-bit block format (kQ4TileBytes tiles, tile-major).
cudaError_t launch_init_weight_q4(uint8_t* dst, int mode, int rows_phys, int cols, int logical_rows, uint64_t seed,
                                  uint64_t tid0, int qd, int kvd, int hd, cudaStream_t st);
cudaError_t launch_init_kv_random(__nv_bfloat16* cache, int B, int H, int hd, int cap, int P, int layer,
                                  int which, int L, uint64_t seed, cudaStream_t st);
// x = embedding rows of the window's ids (fp32), xb = bf16(x), sq[d/128][N] = per-128-feature
// sums of x^2, cur[N] = the ids (for the LM head's current-token probability).
// T rows per sequence: the first Tw at the window positions seq_kv[b] + t, the rest at the
// prefix positions trk[b (T - Tw) + t - Tw] (< 0: id 0).
cudaError_t launch_embed(const int* tok, int tok_ld, const int* seq_kv, const __nv_bfloat16* emb, float* x,
                         __nv_bfloat16* xb, float* sq, int* cur, int* epoch, int B, int T, int d, cudaStream_t st,
                         int Tw = -1, const int* trk = nullptr);
// Sparse cache refresh: trk[b R + r] = the r-th COMMITTED position of sequence b below
// seq_kv[b] (ascending), -1 past the last (state rows st + b ld); merge: the K/V rows of the
// refreshed positions (merge[b R + r] != 0) from the side buffers [L][2][B][H][R][hd] into the
// cache [L][2][kv_B][H][cap][hd] (H: the K/V heads).
cudaError_t launch_scr_select(const uint8_t* st, int ld, const int* seq_kv, int* trk, int B, int R,
                              cudaStream_t stream);
cudaError_t launch_scr_merge(const __nv_bfloat16* side, __nv_bfloat16* cache, const int* trk, const int* merge, int L,
                             int B, int kv_B, int H, int hd, int cap, int R, cudaStream_t stream);
// The kernels below are launched with PDL when `pdl` (inside the context's step chain); the
// single-kernel entry points pass false because their inputs may come from foreign kernels.
// Attention plan: CTAs (split, head, sequence x query tile of 16*nw rows); the csize
// splits of one (sequence, head, query tile) form a thread-block cluster and merge
// their partials through distributed shared memory.
struct AttnPlan {
    int qtiles, nw, csize;
    int nb;     // K/V sub-blocks in flight per CTA (1 or 2)
    int pairs;  // warp groups per CTA, each on its own share of the CTA's sub-blocks (1 or 2)
    bool tc;    // head dim 128: the tcgen05 kernel (128-row query tiles, 64-key sub-blocks)
    int qx;     // the last qx of a sequence's T rows are queries only: keys = kv_len + T - qx
};
// Finer ordering of the mma.sync attention after the chained projections that computed its
// q/K/V (null: the whole preceding grid, by griddepcontrol.wait).  The attention of a
// (sequence, head) starts once the QKV phase has published the tiles holding query head h's
// rows, K head hk's and V head hk's for the sequence's token columns; before it exits, the
// CTA still waits for the whole preceding grid, so a kernel ordered after the attention by
// griddepcontrol.wait stays ordered after that grid too.
struct AttnSync {
    const int* qkv_done;  // the QKV phase's tile flags, [m-tile][token tile]
    int qkv_ntile;        // token columns per token tile
    int qkv_ntiles;       // token tiles
    int k_row0, v_row0;   // first K row, first V row of the fused QKV output
    const int* epoch;     // the flags' tag: *epoch * tag_mul + tag_add (the chain's tagging)
    int tag_mul, tag_add;
};
// head dim 128 and at least kTcMinKeys keys: the tcgen05 kernel's plan; otherwise the
// mma.sync kernel's
constexpr int kTcMinKeys = 1024;
AttnPlan attn_plan(int B, int T, int H, int hd, int max_keys, int sms);
AttnPlan attn_plan_tc(int B, int T, int H, int max_keys, int sms);
cudaError_t attn_tc_init_attrs();
// Grouped-query attention: query head h reads K/V head h / (H / Hkv) of the cache [B][Hkv][cap][hd].
cudaError_t launch_attention_tc(const __nv_bfloat16* q, const __nv_bfloat16* kc, const __nv_bfloat16* vc,
                                const int* seq_kv, __nv_bfloat16* out, int B, int T, int H, int Hkv, int cap,
                                const AttnPlan& a, cudaStream_t st, bool pdl, unsigned long long* trace,
                                int* status);
cudaError_t launch_attention(const __nv_bfloat16* q, const __nv_bfloat16* kc, const __nv_bfloat16* vc,
                             const int* seq_kv, __nv_bfloat16* out, int B, int T, int H, int Hkv, int hd, int cap,
                             const AttnPlan& a, cudaStream_t st, bool pdl = true,
                             unsigned long long* trace = nullptr, int* status = nullptr,
                             const AttnSync* sync = nullptr);
cudaError_t launch_lmhead_reduce(const float* lm_part, const float* zcur, const int* cur_tok, int m_tiles,
                                 int N, int mask_id, int* x0, float* conf, float* tokconf, cudaStream_t st,
                                 bool pdl = true, const int* row_map = nullptr, const int* n_rows = nullptr);
// Selective logits skipping (Sec. 3.3): the rows of the step that need a decision are those whose
// position is MASKED, COMMITTED or DRAFT (tracked refresh rows always); FIXED and STABLE rows
// skip the LM head.  launch_sls_map (one CTA) lists the needed rows in ascending order
// (row_map[0..*n_rows)) and gives every skipped row the decision x0 = -1, conf = tokconf = 0;
// launch_sls_gather copies the listed rows' bf16 activations, RMSNorm statistics and current
// ids into compact buffers and zero-fills the rest of the last token tile (pad_to rows).
cudaError_t launch_sls_map(const uint8_t* st, int ld, const int* seq_kv, int use_cache, int B, int Tw, int T,
                           int* row_map, int* n_rows, int* x0, float* conf, float* tokconf, cudaStream_t stream);
cudaError_t launch_sls_gather(const int* row_map, const int* n_rows, int N, int pad_to, int d,
                              const __nv_bfloat16* xn, const float* sq, int n_sq, const int* cur,
                              __nv_bfloat16* xc, float* sqc, int* curc, cudaStream_t stream);

// Commit pass.  Per sequence b: state arrays at tok + b*ld, st + b*ld; the
// window starts at seq_kv[b] (prefix cache on) or 0 (off); plan[b] holds
// {c0, c1, step}.
struct CommitArgs {
    int* tok;
    uint8_t* st;
    int ld;
    const int* seq_kv;
    int* plan;           // [B][4]: c0, c1, step, spare
    const int* x0;       // [B][T] window-indexed
    const float* conf;
    const float* tokconf;
    int* outs;           // [B][8]: committed, remasked, stable, drafts, done, masked_after
    int* slide_kv;       // continuous sliding: the per-sequence cache frontier to advance (null: off)
    int B, T, mask_id, use_cache;
    int S, remask_max, spec_blocks, block_len;
    float theta_remask, theta_stable;
    int commit_mode;     // DLLM_COMMIT_SCHEDULE / DLLM_COMMIT_THRESHOLD (dllm.h)
    float theta_visible;
    // rows per sequence of x0 / conf / tokconf (T, or T + R with sparse cache refresh: row
    // T + r of sequence b is the prefix position trk[b R + r]); merge[b R + r]: its K/V are merged
    int Tq, R;
    const int* trk;
    int* merge;
};
cudaError_t launch_commit(const CommitArgs& a, cudaStream_t st, bool pdl = true);

cudaError_t launch_begin_block(int* tok, uint8_t* st, int* snap_tok, uint8_t* snap_st, int ld, int n_pos, int* plan,
                               int B, int c0, int c1, cudaStream_t stream);
cudaError_t launch_rewind(int* tok, uint8_t* st, const int* snap_tok, const uint8_t* snap_st, int ld, int n_pos,
                          int* plan, int B, cudaStream_t stream);
cudaError_t launch_set_kv_len(int* seq_kv, int B, int v, cudaStream_t stream);
cudaError_t gemm_init_attrs();
cudaError_t attn_init_attrs();

}  // namespace dllm
