/*
 * dllm_ops.h - single-kernel entry points of the denoising path, for
 * kernel-level parity tests and micro-benchmarks.  Same conventions as
 * dllm.h (0 = OK, negative DLLM_E* codes; messages via dllm_last_error(NULL)).
 * Device pointers are marked "dev"; these calls allocate their own scratch
 * with cudaMalloc and free it before returning, and synchronise the stream.
 */
#ifndef DLLM_OPS_H
#define DLLM_OPS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Dense projection of the transformer step (Sec. 2.1, the matrix work the
 * paper offloads to the NPU; here tcgen05 tensor cores):
 * D[n][m] = sum_k W[m][k] * X[n][k].  W dev bf16 [M][K] row-major, X dev bf16
 * [N][K] row-major, D dev fp32 [N][M].  K*2 bytes must be a multiple of 16;
 * W and X 16-byte aligned.  grid = CTAs of the stream-K split (0 or more
 * than the SM count: one per SM; the CTAs that finish a split tile wait for
 * its other contributors, so all of them must be resident at once).
 * Errors: DLLM_EINVAL, DLLM_ECUDA, DLLM_ETIMEOUT. */
int dllm_op_gemm(const void* W, const void* X, float* D, int M, int N, int K, int grid, void* stream);

/* dllm_op_gemm launched `reps` times back to back on one scratch
 * allocation; *ms_per_launch = average kernel time by CUDA events on the
 * stream (micro-benchmark hook).  flags bit 0: chain the timed launches with
 * programmatic dependent launch; bit 1: plan 227 KB of shared memory instead
 * of 113 KB (one CTA per SM) for <= 96 tokens; bit 2: the bounded-wait test:
 * a single launch whose operand producer waits for a device word that nothing
 * writes, so the wait runs out after about 2 s, every role of the kernel
 * unwinds and the call returns DLLM_ETIMEOUT (ms_per_launch is not set). */
int dllm_op_gemm_timed(const void* W, const void* X, float* D, int M, int N, int K, int grid, int reps, int flags,
                       float* ms_per_launch, void* stream);

/* dllm_op_gemm_timed that also returns a timeline of the last launch:
 * trace [grid_used][16] holds, per CTA, %globaltimer stamps (ns) at entry,
 * after the prologue, first operand stage arrived, last stage consumed,
 * epilogue done, exit; the SM id; the stamp when the dependency wait
 * returned; for the CTA's last output tile: accumulator ready, split partial
 * stored (or, for the CTA that finishes the tile, its wait started), all
 * contributors arrived and partials reduced (0 unless this CTA finishes the
 * tile), the finishing flag and the tile index.  trace must hold 16 values
 * per SM. */
int dllm_op_gemm_trace(const void* W, const void* X, float* D, int M, int N, int K, int grid, int reps,
                       float* ms_per_launch, unsigned long long* trace, int* grid_used, void* stream);

/* dllm_op_gemm for callers that cannot allocate device memory.  Such callers
 * exist: an application (a serving engine, a game, a plugin host) often hands
 * nearly all of a GPU's memory to its own pool allocator at start-up, so a
 * cudaMalloc from a library it calls fails or breaks its accounting, and a
 * latency-critical loop cannot afford the implicit device synchronisation
 * that cudaMalloc and cudaFree may cause.  The paper has no counterpart: this
 * is a property of this library's API.
 * It computes the same D[n][m] = sum_k W[m][k] * X[n][k] as dllm_op_gemm
 * (same arguments, same layouts) but keeps its scratch (split partials, tile
 * tickets, status word) in one statically sized device array of 8 MiB that
 * every GPU loading the library holds until the process exits; it calls no
 * cudaMalloc, cudaFree or other allocating routine.
 * Limits: at most 2046 output tiles (ceil(M/128) x token tiles of <= 256
 * tokens), else DLLM_ECAPACITY; the grid (0 = one CTA per SM, at most the SM
 * count) is shrunk to fit the array when chosen automatically (for 256-token
 * tiles: 62 CTAs), and an explicit grid that does not fit is rejected with
 * DLLM_ECAPACITY.
 * The first call on a device looks up the array's device address
 * (cudaGetSymbolAddress) with that device current.  Every call shares the
 * one array and clears its tickets and status word before its launch: two
 * calls that overlap on the GPU (other streams, other host threads) race and
 * corrupt each other's results.  Synchronises the stream.
 * Errors: DLLM_EINVAL, DLLM_ECAPACITY, DLLM_ECUDA, DLLM_ETIMEOUT. */
int dllm_op_gemm_noalloc(const void* W, const void* X, float* D, int M, int N, int K, int grid, void* stream);

/* Bidirectional attention of the window's queries over cached + window keys
 * (Sec. 2.1, block-wise decoding with prefix KV reuse; no causal mask).
 * q dev bf16 [B][H][T][hd]; kc, vc dev bf16 [B][Hkv][cap][hd] (keys of
 * sequence b: positions [0, kv_len[b] + T)); kv_len dev int32 [B];
 * out dev bf16 [B*T][H*hd].  hd in {64, 128}.  Hkv = H is multi-head
 * attention; Hkv < H (dividing H) is grouped-query attention (the Dream-7B
 * model of Sec. 5.1): query head h reads K/V head h / (H / Hkv). */
int dllm_op_attention(const void* q, const void* kc, const void* vc, const int32_t* kv_len, void* out, int B, int T,
                      int H, int Hkv, int hd, int cap, int max_kv_len, void* stream);

/* LM head with decision (Sec. 2.1 confidence-selected commits; Sec. 3.3
 * selective logits): per token n, z = W X[n]^T over the vocab; x0 = argmax
 * excluding mask_id (ties: lowest id); conf = softmax(z)[x0] with the mask
 * excluded; tokconf = softmax(z)[cur[n]] (0 when cur[n] is the mask id).
 * W dev bf16 [V][d], X dev bf16 [N][d], cur dev int32 [N]; outputs dev [N];
 * logits dev fp32 [N][V] or NULL. */
int dllm_op_lmhead(const void* W, const void* X, const int32_t* cur, int32_t* x0, float* conf, float* tokconf,
                   float* logits, int V, int N, int d, int mask_id, void* stream);

/* One commit / re-mask / draft pass on HOST arrays of one sequence
 * (Sec. 2.1 commit, Sec. 3.2 drafts, Sec. 3.3 revision and staged token
 * stabilization; commit_mode / theta_visible as in dllm_sched): tok int32 and
 * status uint8 [n_pos] are updated in place; x0, conf, tokconf [T] are
 * indexed by window offset; window [w0, w0+T), current block [c0, c1),
 * step index within the block.  sched as in dllm.h; block_len = draft block
 * size.  out nullable.  Runs the device kernel on copies. */
int dllm_op_commit(int32_t* tok, uint8_t* status, int n_pos, int w0, int T, int c0, int c1, int step,
                   const int32_t* x0, const float* conf, const float* tokconf, int steps_per_block,
                   float theta_remask, float theta_stable, int remask_max, int spec_blocks, int use_prefix_cache,
                   int block_len, int mask_id, int commit_mode, float theta_visible, int* out6);

#ifdef __cplusplus
}
#endif
#endif
