// dllm_op_gemm_noalloc: the tensor-core projection of dllm_op_gemm for callers
// that must not allocate device memory.
//
// Its scratch (the stream-K split partials, the per-tile tickets and the status
// word) lives in one file-scope __device__ array of kNoAllocScratchBytes, which
// every GPU that loads this library holds until the process exits.  Host code
// cannot use the array's name as a device address (in host code the symbol is
// a host-side stand-in), so the first call on each device looks up the real
// address with cudaGetSymbolAddress while that device is current, and keeps it.
// The mutex below covers only that one-time lookup: the calls themselves share
// the array without any ordering, so two calls that overlap on the GPU race.
#include "../../include/dllm.h"
#include "../../include/dllm_ops.h"
#include "internal.h"

#include <mutex>

using namespace dllm;

void dllm_set_noctx_error(const char* msg);

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(8) << 20;   // 8 MiB per GPU
constexpr size_t kTicketBytes = 256 << 10;                 // tickets + status word at the front
constexpr int kMaxTickets = (kTicketBytes - 256) / 128;    // tiles x token tiles, one per 128-byte line
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_gemm_scratch[kNoAllocScratchBytes];

std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

int noalloc_fail(int code, const char* msg) {
    dllm_set_noctx_error(msg);
    return code;
}

// Device address of g_gemm_scratch on the current device (looked up once).
int scratch_address(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return noalloc_fail(DLLM_ECUDA, "no usable CUDA device");
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_gemm_scratch);
        if (e != cudaSuccess || !p) return noalloc_fail(DLLM_ECUDA, cudaGetErrorString(e));
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return DLLM_OK;
}

}  // namespace

extern "C" int dllm_op_gemm_noalloc(const void* W, const void* X, float* D, int M, int N, int K, int grid,
                                    void* stream) {
    if (!W || !X || !D || M < 1 || N < 1 || K < 1 || (K * 2) % 16 || grid < 0)
        return noalloc_fail(DLLM_EINVAL, "bad gemm arguments");
    void* base = nullptr;
    int rc = scratch_address(&base);
    if (rc) return rc;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
        return noalloc_fail(DLLM_ECUDA, "device query failed");
    GemmPlan p = gemm_plan(M, N, K, (grid > 0 && grid < sms) ? grid : sms, EPI_F32);
    p.pdl = false;
    // the split partials sit behind the tickets; gemm_partial_floats is the bound gemm_launch
    // checks, so the grid that fits is the one whose partials fit the rest of the array
    GemmPlan one = p;
    one.grid = 1;
    const size_t per_cta = gemm_partial_floats(one) * sizeof(float);
    const size_t cap_ctas = (kNoAllocScratchBytes - kTicketBytes) / per_cta;
    if (static_cast<long long>(p.m_tiles) * p.n_tiles > kMaxTickets)
        return noalloc_fail(DLLM_ECAPACITY, "too many output tiles for the static scratch (M x N too large)");
    if (static_cast<size_t>(p.grid) > cap_ctas) {
        if (grid > 0) return noalloc_fail(DLLM_ECAPACITY, "grid too large for the static scratch");
        p = gemm_plan(M, N, K, static_cast<int>(cap_ctas), EPI_F32);  // auto grid: shrink to fit
        p.pdl = false;
    }
    if (gemm_init_attrs() != cudaSuccess) return noalloc_fail(DLLM_ECUDA, "attribute setup failed");
    CUtensorMap tw, tx;
    if (!make_tmap_bf16(&tw, W, M, K, 128) || !make_tmap_bf16(&tx, X, N, K, p.ntile))
        return noalloc_fail(DLLM_EINVAL, "tensor map encode failed (alignment?)");
    unsigned char* s = static_cast<unsigned char*>(base);
    int* tickets = reinterpret_cast<int*>(s + 256);
    int* status = reinterpret_cast<int*>(s);
    float* partials = reinterpret_cast<float*>(s + kTicketBytes);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // the array keeps the previous call's contents: start tickets and status at zero
    if (cudaMemsetAsync(s, 0, kTicketBytes, st) != cudaSuccess) return noalloc_fail(DLLM_ECUDA, "memset failed");
    Scratch scr{partials, tickets, (kNoAllocScratchBytes - kTicketBytes) / sizeof(float), kMaxTickets * 32};
    EpiArgs ep{};
    ep.out = D;
    ep.ld_out = M;
    cudaError_t e = gemm_launch(EPI_F32, p, tw, tx, ep, scr, status, st);
    if (e != cudaSuccess) return noalloc_fail(DLLM_ECUDA, cudaGetErrorString(e));
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return noalloc_fail(DLLM_ECUDA, cudaGetErrorString(e));
    int sv = 0;
    if (cudaMemcpy(&sv, status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
        return noalloc_fail(DLLM_ECUDA, "status read failed");
    if (sv & kStatusTimeout) return noalloc_fail(DLLM_ETIMEOUT, "bounded device wait ran out");
    if (sv) return noalloc_fail(DLLM_ECUDA, "device status error");
    return DLLM_OK;
}
