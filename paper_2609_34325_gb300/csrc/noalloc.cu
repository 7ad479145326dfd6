// dora_pruned_block_noalloc: the pruned block with its scratch memory held by
// the library itself, for callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocating routine) at the
// point where they run the block: code on a path that must never
// synchronise the device (cudaMalloc and cudaFree may synchronise), plugins
// whose host framework owns every byte of device memory through its own pool
// and forbids side allocations, or processes that reserved the whole device
// up front.  This entry point lets them run a block by passing only inputs
// and outputs: the intermediates live in the file-scope array below.
//
// Cost: every GPU that loads the library holds kScratchBytes of device memory
// for the scratch array until the process exits.
#include <cuda_runtime.h>
#include <stdint.h>

#include <mutex>

#include "dora.h"

namespace {

constexpr size_t kScratchBytes = DORA_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

// The block's workspace.  In host code this name is only a stand-in for the
// symbol; the device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) uint8_t g_block_scratch[kScratchBytes];

std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices];   // device address of g_block_scratch per device

// Set-up, once per device, with that device current: look up the device
// address of the scratch array.  Returns nullptr on failure.
void* scratch_for_current_device() {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_block_scratch) != cudaSuccess || p == nullptr) {
      cudaGetLastError();
      return nullptr;
    }
    g_scratch_addr[dev] = p;
  }
  return g_scratch_addr[dev];
}

}  // namespace

extern "C" int dora_pruned_block_noalloc(const dora_bf16* x_in, const int32_t* cu_in,
                                         const int32_t* ids_in, int32_t batch,
                                         int32_t max_seqlen, int32_t t_cap,
                                         const dora_block_weights* w, const float* scores,
                                         const int32_t* keep_counts, dora_bf16* x_out,
                                         int32_t* cu_out, int32_t* ids_out, int32_t* kept_idx,
                                         const float* x_in_moments, float* x_out_moments,
                                         int32_t* status, dora_stream_t stream) {
  if (w == nullptr || t_cap < 0 || batch < 0) return DORA_ERR_INVALID_ARG;
  const size_t need = dora_workspace_size(t_cap, batch, w);
  if (need == 0) return DORA_ERR_INVALID_ARG;
  if (need > kScratchBytes) return DORA_ERR_SCRATCH_TOO_SMALL;
  void* scratch = scratch_for_current_device();
  if (scratch == nullptr) return DORA_ERR_CUDA;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // The status word at the start of the scratch must start each call at zero
  // (first error wins); the rest is written before it is read.
  if (cudaMemsetAsync(scratch, 0, sizeof(int32_t), s) != cudaSuccess) return DORA_ERR_CUDA;
  const int rc = dora_pruned_block(x_in, cu_in, ids_in, batch, max_seqlen, t_cap, w, scores,
                                   keep_counts, x_out, cu_out, ids_out, kept_idx, x_in_moments,
                                   x_out_moments, scratch, kScratchBytes, stream);
  if (rc != DORA_OK) return rc;
  if (status != nullptr &&
      cudaMemcpyAsync(status, dora_workspace_status(scratch), sizeof(int32_t),
                      cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return DORA_ERR_CUDA;
  return DORA_OK;
}
