// aal_accept_reward_noalloc: the acceptance reward with its scratch in a fixed device array.
//
// Some callers cannot allocate device memory for a workspace: a training loop whose
// device memory is all reserved up front by its own caching allocator (a raw
// cudaMalloc there fails or fragments that pool), or a host component that only
// receives device pointers from another component and has no allocator of its own.
// This entry point serves them.  Its scratch (the reward workspace: header, per-row
// accept flags, per-window rewards) lives in the file-scope array below, which every
// GPU that loads libaal holds until the process exits.  Nothing is allocated or freed.
#include <mutex>

#include "aal_internal.cuh"

namespace {

constexpr int64_t kNoAllocMaxRows = int64_t(1) << 20;  // N * K logit rows
constexpr size_t kScratchBytes = (size_t(6) << 20) + 4096;  // header + 2 x R flags + 4 N rewards

static __device__ __align__(256) unsigned char g_reward_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
void* g_scratch[kMaxDevices] = {};        // device address of g_reward_scratch, per device
cudaError_t g_setup[kMaxDevices] = {};    // result of the one-time lookup
bool g_tried[kMaxDevices] = {};

// Device address of the scratch array on the current device, looked up once per device.
aal_status scratch_address(void** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return AAL_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mutex);
  if (!g_tried[dev]) {
    void* p = nullptr;
    g_setup[dev] = cudaGetSymbolAddress(&p, g_reward_scratch);
    g_scratch[dev] = p;
    g_tried[dev] = true;
  }
  if (g_setup[dev] != cudaSuccess || g_scratch[dev] == nullptr) return AAL_ERR_CUDA;
  *out = g_scratch[dev];
  return AAL_OK;
}

}  // namespace

extern "C" AAL_API aal_status aal_accept_reward_noalloc(const aal_reward_problem* prob, const void* draft,
                                                        const void* target, const void* ref_draft,
                                                        int32_t* tau, int32_t* tau_ref, float* rollout_len,
                                                        float* advantage, void* stream) {
  size_t need = 0;
  aal_status st = aal_reward_workspace_size(prob, &need);  // validates the problem
  if (st != AAL_OK) return st;
  if (prob->N * prob->K > kNoAllocMaxRows || need > kScratchBytes) return AAL_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  st = scratch_address(&scratch);
  if (st != AAL_OK) return st;
  return aal_accept_reward(prob, draft, target, ref_draft, scratch, kScratchBytes, tau, tau_ref, rollout_len,
                           advantage, stream);
}
