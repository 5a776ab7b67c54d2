// track_disagreement_static: the disagreement score of track_disagreement with
// its scratch held in a fixed device array of this library instead of memory
// the library allocates.
//
// Callers that cannot allocate device memory while they run - a serving process
// whose device memory is entirely reserved up front by its own pool, so that a
// cudaMalloc in mid-run could fail, or a latency-critical loop that cannot take
// the device-wide synchronization a cudaMalloc/cudaFree implies - use this entry
// point.  It allocates nothing: the per-block partial sums live in
// g_dis_scratch below, which every GPU that loads the library holds until the
// process exits.
#include <cuda_runtime.h>

#include <mutex>
#include <string>

#include "../../include/track.h"
#include "internal.h"

namespace track {
namespace {

// Maximum scratch: TRACK_STATIC_MAX_SAMPLES samples x TRACK_STATIC_MAX_BLOCKS
// partial blocks x 2 partial sums = 64 x 512 x 2 floats = 256 KiB per device.
constexpr int kMaxBlocks = TRACK_STATIC_MAX_BLOCKS;
constexpr int kMaxSamples = TRACK_STATIC_MAX_SAMPLES;
__device__ __align__(256) float g_dis_scratch[kMaxSamples * kMaxBlocks * 2];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
float* g_scratch_ptr[kMaxDevices] = {};  // device address of g_dis_scratch, per device

int err(int code, const std::string& msg) {
  return report_error(code, ("track_disagreement_static: " + msg).c_str());
}

}  // namespace
}  // namespace track

using namespace track;

extern "C" int track_disagreement_static(const float* v_L, const float* v_S, int B,
                                         int64_t n_per_sample, float eps, float* score_accum,
                                         track_stream s) {
  if (!v_L || !v_S || !score_accum || B < 0 || n_per_sample <= 0 || !(eps > 0.f))
    return err(TRACK_EINVAL, "bad arguments");
  if (B > kMaxSamples)
    return err(TRACK_EINVAL, "B = " + std::to_string(B) + " exceeds the maximum of " +
                                 std::to_string(kMaxSamples) + " samples per call");
  if (B == 0) return TRACK_OK;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return err(TRACK_ECUDA, "no usable current device");
  // The array's address is per device: a stream of another device would be
  // handed this device's copy.
  if (s != nullptr) {
    int sdev = -1;
    cudaError_t e = cudaStreamGetDevice((cudaStream_t)s, &sdev);
    if (e != cudaSuccess) return err(TRACK_EINVAL, std::string("bad stream: ") + cudaGetErrorString(e));
    if (sdev != dev)
      return err(TRACK_EINVAL, "the stream belongs to device " + std::to_string(sdev) +
                                   ", not to the current device " + std::to_string(dev));
  }
  float* scratch = nullptr;
  {
    // One-time set-up per device, with that device current: the host-side name
    // g_dis_scratch is only a stand-in, so its device address is looked up here.
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_scratch_ptr[dev] == nullptr) {
      void* p = nullptr;
      cudaError_t e = cudaGetSymbolAddress(&p, g_dis_scratch);
      if (e != cudaSuccess) return err(TRACK_ECUDA, std::string("cudaGetSymbolAddress: ") +
                                                      cudaGetErrorString(e));
      g_scratch_ptr[dev] = (float*)p;
    }
    scratch = g_scratch_ptr[dev];
  }
  // Same partition as track_disagreement (so both give the same bits), capped
  // by the array's size.
  int64_t nblk = disagreement_blocks(n_per_sample, B);
  if (nblk > kMaxBlocks) nblk = kMaxBlocks;
  // Every partial slot the reduction reads is written earlier in the same call,
  // so nothing needs clearing between calls.
  cudaError_t e = disagreement(v_L, v_S, B, n_per_sample, eps, score_accum, scratch, (int)nblk,
                               (cudaStream_t)s);
  if (e != cudaSuccess) return err(TRACK_ECUDA, std::string("launch: ") + cudaGetErrorString(e));
  return TRACK_OK;
}
