// dblast_target_lse_noalloc: the target log-sum-exp pass without any device
// allocation, for callers that cannot allocate device memory when they call
// in.  Examples are a plugin running inside another engine's enqueue step and
// code with a fixed device-memory budget.  Such code must not call
// cudaMalloc: the call synchronises the device and bypasses the host engine's
// memory pool, and the caller may not be able to hand out a workspace.
//
// The only scratch is the file-scope array below: one 8-byte record
// (max, sum) per (vocabulary tile of 128, row).  Every GPU that loads the
// library holds it (8 MiB) until the process exits.  Every record the merge
// kernel reads was written earlier in the same call, so nothing has to be
// cleared between calls; calls whose kernels overlap on the GPU (two streams,
// or two threads) share the array and race.
#include <mutex>

#include "dblast_internal.cuh"

namespace dblast {

constexpr unsigned kNoAllocRecords = DBLAST_NOALLOC_MAX_RECORDS;
static __device__ __align__(256) float2 g_noalloc_scratch[kNoAllocRecords];

// one warp per (row, tile): (m2, s) of the tile's t / T in base 2
template <typename Tin>
__global__ void k_noalloc_tiles(const Tin* __restrict__ target, int rows, int V, int nt, float k2,
                                float2* __restrict__ rec) {
  const long long gw = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (gw >= (long long)rows * nt) return;
  const int row = (int)(gw / nt), t = (int)(gw - (long long)row * nt);
  const Tin* tr = target + (size_t)row * V;
  float s[4];
  float mx = -INFINITY;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int v = t * TILE_V + lane * 4 + j;
    s[j] = (v < V) ? ldf(tr + v) * k2 : -INFINITY;
    mx = fmaxf(mx, s[j]);
  }
  float2 p = make_float2(-INFINITY, 0.f);
  if (mx != -INFINITY) {
    float sum = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) sum += (s[j] != -INFINITY) ? exp2f(s[j] - mx) : 0.f;
    p = make_float2(mx, sum);
  }
  p = warp_lse_merge(p);
  if (lane == 0) rec[(size_t)t * rows + row] = p;
}

// one warp per row: merge the row's records, natural-log result
__global__ void k_noalloc_merge(const float2* __restrict__ rec, int rows, int nt,
                                float* __restrict__ lse_out) {
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (row >= rows) return;
  float mx = -INFINITY;
  for (int t = lane; t < nt; t += 32) mx = fmaxf(mx, rec[(size_t)t * rows + row].x);
  mx = warp_max(mx);
  double s = 0.0;
  if (mx != -INFINITY)
    for (int t = lane; t < nt; t += 32) {
      const float2 q = rec[(size_t)t * rows + row];
      if (q.y > 0.f) s += (double)q.y * exp2((double)q.x - (double)mx);
    }
  s = warp_sum_d(s);
  if (lane == 0)
    lse_out[row] = mx == -INFINITY ? -INFINITY : (float)(((double)mx + log2(s)) * (double)LN2);
}

// Device address of the static scratch, looked up once per device with that
// device current (the first call on each device does it), and again when the
// device's context has changed since (a cudaDeviceReset loads the library's
// device code anew, at an address that may differ).
static std::mutex g_noalloc_mu;
static float2* g_noalloc_addr[128] = {};
static unsigned long long g_noalloc_ctx[128] = {};

static cudaError_t noalloc_scratch(float2** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 128) return cudaErrorInvalidDevice;
  const unsigned long long ctx = current_context_id();
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_addr[dev] || g_noalloc_ctx[dev] != ctx) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_noalloc_addr[dev] = static_cast<float2*>(p);
    g_noalloc_ctx[dev] = ctx;
  }
  *out = g_noalloc_addr[dev];
  return cudaSuccess;
}

}  // namespace dblast

using namespace dblast;

extern "C" dblast_status dblast_target_lse_noalloc(const void* target, int rows, int V,
                                                   dblast_dtype dtype, float temperature,
                                                   float* lse_out, dblast_stream_t stream) {
  if (!target || !lse_out || rows < 1 || V < 1 || !(temperature > 0.f) ||
      (dtype != DBLAST_BF16 && dtype != DBLAST_F32))
    return DBLAST_ERR_INVALID_ARG;
  const int nt = ceil_div(V, TILE_V);
  if ((unsigned long long)rows * (unsigned long long)nt > kNoAllocRecords)
    return DBLAST_ERR_WORKSPACE;  // rows * ceil(V/128) exceeds the static scratch
  float2* rec = nullptr;
  cudaError_t e = noalloc_scratch(&rec);
  if (e != cudaSuccess) return DBLAST_ERR_CUDA;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const float k2 = LOG2E / temperature;
  const unsigned blocks = (unsigned)(((long long)rows * nt * 32 + 255) / 256);
  if (dtype == DBLAST_F32)
    k_noalloc_tiles<float><<<blocks, 256, 0, s>>>(static_cast<const float*>(target), rows, V,
                                                   nt, k2, rec);
  else
    k_noalloc_tiles<__nv_bfloat16><<<blocks, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(target), rows, V, nt, k2, rec);
  k_noalloc_merge<<<ceil_div(rows * 32, 256), 256, 0, s>>>(rec, rows, nt, lse_out);
  e = cudaGetLastError();
  return e == cudaSuccess ? DBLAST_OK : DBLAST_ERR_CUDA;
}
