// turnopd_loss_fwd_bwd_static: the loss entry point with its scratch space in
// a file-scope device array, for callers that cannot allocate device memory.
// It forwards to turnopd_loss_fwd_bwd with that array as the workspace.

#include <atomic>

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
std::atomic<void *> g_scratch_addr[kMaxDevices];

// Device address of g_loss_scratch on the current device (looked up once per
// device; the host-side symbol itself is not a device address).
turnopd_status scratch_address(void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return TURNOPD_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices)
        return TURNOPD_ERR_UNSUPPORTED;
    void *p = g_scratch_addr[dev].load(std::memory_order_acquire);
    if (!p) {
        if (cudaGetSymbolAddress(&p, g_loss_scratch) != cudaSuccess || !p)
            return TURNOPD_ERR_CUDA;
        g_scratch_addr[dev].store(p, std::memory_order_release);
    }
    *out = p;
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
