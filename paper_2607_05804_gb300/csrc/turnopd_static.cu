// turnopd_loss_fwd_bwd_static: the loss entry point with its scratch space in
// a file-scope device array, for callers that cannot allocate device memory.
// It forwards to turnopd_loss_fwd_bwd with that array as the workspace.

#include <mutex>

#include <cuda.h>

#include "common.cuh"
#include "kernels.h"

namespace {

// Same layout as the loss workspace for TURNOPD_STATIC_MAX_TOKENS tokens:
// row records (16 B/token), per-block counts, the row count, w*l per row (8 B/token).
constexpr size_t a256(size_t x) { return (x + 255) & ~size_t(255); }
constexpr size_t kTokens = TURNOPD_STATIC_MAX_TOKENS;
constexpr size_t kBlocks = (kTokens + turnopd::kCompactBlock - 1) / turnopd::kCompactBlock;
constexpr size_t kBytes = a256(16 * kTokens) + a256(4 * (kBlocks + 1)) + a256(4) + a256(8 * kTokens) + 256;
static_assert(kBytes == TURNOPD_STATIC_SCRATCH_BYTES, "header constant out of date");

// Shared by every call on a device; held until the process exits.
static __device__ __align__(256) unsigned char g_loss_scratch[kBytes];

constexpr int kMaxDevices = 64;

// The array's device address belongs to one CUDA context: after a
// cudaDeviceReset (or any teardown of the primary context) the module is
// loaded again and the array may sit elsewhere.  So the cached address is
// keyed on the context's process-unique id (cuCtxGetId), and looked up again
// whenever the current context is not the one it was taken in.
struct ScratchSlot {
    std::mutex mu;
    unsigned long long ctx_id = 0;
    void *addr = nullptr;
};
ScratchSlot g_slot[kMaxDevices];

typedef CUresult (*PFN_ctxGetCurrent)(CUcontext *);
typedef CUresult (*PFN_ctxGetId)(CUcontext, unsigned long long *);

template <class F>
F driver_fn(const char *name, int version)
{
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion(name, &p, version, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
        return nullptr;
    return reinterpret_cast<F>(p);
}

// Id of the context current on this thread (0 if none is current yet).
turnopd_status current_ctx_id(unsigned long long *id)
{
    static PFN_ctxGetCurrent get_current = driver_fn<PFN_ctxGetCurrent>("cuCtxGetCurrent", 4000);
    static PFN_ctxGetId get_id = driver_fn<PFN_ctxGetId>("cuCtxGetId", 12000);
    if (!get_current || !get_id)
        return TURNOPD_ERR_CUDA;
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS)
        return TURNOPD_ERR_CUDA;
    *id = 0;
    if (ctx && get_id(ctx, id) != CUDA_SUCCESS)
        return TURNOPD_ERR_CUDA;
    return TURNOPD_OK;
}

// Device address of g_loss_scratch in the current context of the current
// device.  The lookup (cudaGetSymbolAddress, which also makes the runtime's
// primary context current if none is) runs on the first call in a context;
// later calls in the same context take the cached address.
turnopd_status scratch_address(void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return TURNOPD_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices)
        return TURNOPD_ERR_UNSUPPORTED;
    unsigned long long id = 0;
    turnopd_status st = current_ctx_id(&id);
    if (st != TURNOPD_OK)
        return st;
    ScratchSlot &slot = g_slot[dev];
    std::lock_guard<std::mutex> lock(slot.mu);
    if (id == 0 || id != slot.ctx_id || !slot.addr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_loss_scratch) != cudaSuccess || !p)
            return TURNOPD_ERR_CUDA;
        if ((st = current_ctx_id(&id)) != TURNOPD_OK || id == 0)
            return st != TURNOPD_OK ? st : TURNOPD_ERR_CUDA;
        slot.ctx_id = id;
        slot.addr = p;
    }
    *out = slot.addr;
    return TURNOPD_OK;
}

}  // namespace

extern "C" turnopd_status turnopd_loss_fwd_bwd_static(
    const void *z_student, const void *z_teacher, int32_t in_dtype, int64_t ld, int64_t vocab,
    int64_t num_rows, const int32_t *row_of_token, const int32_t *sampled_ids,
    const uint8_t *loss_mask, const float *w, int64_t num_tokens, int32_t mode, void *grad_student,
    int32_t grad_dtype, uint32_t flags, float *token_loss_out, double *loss_out,
    int32_t *dev_status, turnopd_stream_t stream)
{
    if (num_tokens > (int64_t)TURNOPD_STATIC_MAX_TOKENS)
        return TURNOPD_ERR_WORKSPACE;
    if (turnopd::loss_workspace_bytes(num_tokens < 0 ? 0 : num_tokens) > kBytes)
        return TURNOPD_ERR_WORKSPACE;
    void *ws = nullptr;
    turnopd_status st = scratch_address(&ws);
    if (st != TURNOPD_OK)
        return st;
    return turnopd_loss_fwd_bwd(z_student, z_teacher, in_dtype, ld, vocab, num_rows, row_of_token,
                                sampled_ids, loss_mask, w, num_tokens, mode, grad_student,
                                grad_dtype, flags, token_loss_out, loss_out, ws, kBytes,
                                dev_status, stream);
}
