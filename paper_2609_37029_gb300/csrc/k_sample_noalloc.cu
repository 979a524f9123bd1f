// lsp_sample_noalloc: the correction + sampling step for callers that cannot
// allocate device memory.
//
// Some callers of this library cannot call cudaMalloc at the point where they
// sample: a serving loop that runs inside a custom allocator's critical
// section, a process whose device memory is fully reserved by another
// framework's caching allocator, or code that must not create a state object
// (lsp_state_create allocates the interface and a workspace).  The sampler's
// only scratch is the per-CTA argmax partials of two consecutive steps and the
// per-step keys and arrival counters of the persistent kernel, so this variant
// keeps them in a fixed file-scope __device__ array instead.  Every GPU that
// loads the library holds that array until the process exits.  The counters
// are cleared on the caller's stream before every launch, so a launch that
// gave up waiting cannot affect the next one.
#include <cmath>
#include <mutex>

#include "lsp_internal.h"

namespace {

constexpr size_t kStaticScratchBytes = 512 * 1024;     // the documented maximum (512 KiB)
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_sample_scratch[kStaticScratchBytes];

struct DeviceScratch {
  std::mutex mu;
  bool ready = false;               // set only after both lookups succeeded
  unsigned char* ptr = nullptr;     // device address of g_sample_scratch on this device
  int num_sms = 0;
};
DeviceScratch g_dev[kMaxDevices];

// Per device, with that device current: the device address of the array (the
// host-side symbol is only a stand-in) and the SM count.  Only a successful
// lookup is remembered; after a failure (a transient error, or a first call
// made during stream capture) the next call on that device tries again.
int scratch_for_current_device(unsigned char** ptr, int* num_sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return LSP_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return LSP_ERR_UNSUPPORTED;
  DeviceScratch& ds = g_dev[dev];
  std::lock_guard<std::mutex> lock(ds.mu);
  if (!ds.ready) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_sample_scratch) != cudaSuccess) return LSP_ERR_CUDA;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1)
      return LSP_ERR_CUDA;
    ds.ptr = static_cast<unsigned char*>(p);
    ds.num_sms = sms;
    ds.ready = true;
  }
  *ptr = ds.ptr;
  *num_sms = ds.num_sms;
  return LSP_OK;
}

}  // namespace

extern "C" int lsp_sample_noalloc(const float* base_logits, const int32_t* prev_token,
                                  const void* Ec, const void* Wc, int dtype, int C, int B, int V,
                                  int rc, const lsp_sample_params* sp, int32_t* out_tokens,
                                  float* out_logits, uint32_t* dev_error, lsp_stream_t stream) {
  if (!base_logits || !prev_token || !Ec || !Wc || !sp || !out_tokens) return LSP_ERR_ARG;
  if (dtype != LSP_DTYPE_BF16 && dtype != LSP_DTYPE_F32) return LSP_ERR_ARG;
  if (!(sp->temperature >= 0.f) || !std::isfinite(sp->temperature)) return LSP_ERR_ARG;
  if (C < 1 || C > 64 || B < 1 || V < 16 || V % 16 || rc < 16 || rc % 16 || rc > 256)
    return LSP_ERR_SHAPE;
  unsigned char* scratch = nullptr;
  int num_sms = 0;
  const int rc_setup = scratch_for_current_device(&scratch, &num_sms);
  if (rc_setup != LSP_OK) return rc_setup;
  // Layout: argmax partials of two consecutive steps (values, then indices), then the
  // persistent kernel's step keys and arrival counters -- align256(16 nblk C) +
  // sample_sync_bytes(B) bytes, which must fit the array.
  const int nblk = lsp::sample_blocks(num_sms);
  const size_t part = (size_t)2 * nblk * C;
  const size_t sync_off = (part * (sizeof(float) + sizeof(int)) + 255) / 256 * 256;
  const size_t sync_bytes = lsp::sample_sync_bytes(B);
  if (sync_off + sync_bytes > kStaticScratchBytes) return LSP_ERR_SHAPE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaMemsetAsync(scratch + sync_off, 0, sync_bytes, s) != cudaSuccess) return LSP_ERR_CUDA;
  lsp::SampleParams p = {};
  p.src = base_logits;
  p.dst = out_logits;
  p.prev = prev_token;
  p.prev_stride = 1;
  p.Ec = Ec;
  p.Wc = Wc;
  p.out_tokens = out_tokens;
  p.part_val = reinterpret_cast<float*>(scratch);
  p.part_idx = reinterpret_cast<int*>(scratch + part * sizeof(float));
  p.sync = reinterpret_cast<unsigned long long*>(scratch + sync_off);
  p.err = reinterpret_cast<unsigned*>(dev_error);
  p.C = C;
  p.B = B;
  p.V = V;
  p.rc = rc;
  p.nblk = nblk;
  p.num_sms = num_sms;
  p.temperature = sp->temperature;
  p.round = sp->round;
  p.seed = sp->seed;
  return lsp::launch_sample(p, dtype, s);
}
