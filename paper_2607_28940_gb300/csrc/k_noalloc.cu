// Allocation-free attention pooling of the global anchor.
//
// Some callers cannot allocate device memory while they serve: a process that
// reserves all of its GPU memory up front under its own pool and forbids
// driver allocations afterwards, a plugin running inside another runtime that
// gives it no allocator, or a latency-critical path that cannot afford the
// implicit device synchronisation of cudaMalloc/cudaFree.  txs_pool_anchor_static
// serves them: it computes the same pooled anchor g as the cache build, but its
// scratch (per-slice online-softmax states) lives in the file-scope array below,
// which every GPU that loads this library holds until the process exits.
//
// The caller still passes the behavior rows and the output buffer.  The
// library never calls cudaMalloc, cudaFree or any allocating routine here.
#include <string>

#include "txs_internal.cuh"

namespace txs {

void set_last_error(const char* msg);

namespace {

constexpr int kSlots = 16;                        // slices per request
constexpr int kPiece = 128;                       // rows per online-softmax piece
constexpr long long kScratchFloats = 1 << 20;     // 4 MiB of static scratch
constexpr int kMaxReq = 1024;                     // offsets passed by value
constexpr int kMaxD = 512;                        // two accumulator columns per thread of 256

static __device__ __align__(256) float g_anchor_scratch[kScratchFloats];

struct StaticPoolArgs {
  int n_req;
  int d;
  float inv_sqrt_d;
  int off[kMaxReq + 1];
};

// Slice `slot` of request r: rows [beg, end) split into kSlots near-equal
// slices, each reduced in pieces of kPiece rows with a running max.  Writes
// (m, s, acc[d]) of the slice; an empty slice writes (-inf, 0, 0).
template <typename T>
__global__ void __launch_bounds__(256) pool_slices_static_kernel(const __grid_constant__ StaticPoolArgs a,
                                                                 const T* __restrict__ phi,
                                                                 const float* __restrict__ w_pool,
                                                                 float* __restrict__ scratch) {
  __shared__ float z[kPiece];
  __shared__ float red[8];
  const int r = blockIdx.y, slot = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int d = a.d;
  const int rb = a.off[r], re = a.off[r + 1];
  const int span = (re - rb + kSlots - 1) / kSlots;
  const int beg = rb + slot * span;
  const int end = min(re, beg + span);
  float* out = scratch + (static_cast<long long>(r) * kSlots + slot) * (d + 2);
  float m_run = -INFINITY, s_run = 0.f;
  float acc[2] = {0.f, 0.f};   // columns tid and tid + 256 (d <= kMaxD)
  for (int p0 = beg; p0 < end; p0 += kPiece) {
    const int n = min(kPiece, end - p0);
    for (int i = warp; i < n; i += 8) {
      const T* row = phi + static_cast<long long>(p0 + i) * d;
      float dot = 0.f;
      for (int k = lane; k < d; k += 32) dot = fmaf(Elem<T>::load(row + k), __ldg(w_pool + k), dot);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
      if (lane == 0) z[i] = dot * a.inv_sqrt_d;
    }
    __syncthreads();
    float mp = -INFINITY;
    for (int i = tid; i < n; i += 256) mp = fmaxf(mp, z[i]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mp = fmaxf(mp, __shfl_xor_sync(0xffffffffu, mp, o));
    if (lane == 0) red[warp] = mp;
    __syncthreads();
    mp = red[0];
#pragma unroll
    for (int w = 1; w < 8; ++w) mp = fmaxf(mp, red[w]);
    const float m_new = fmaxf(m_run, mp);
    const float scale_old = expf(m_run - m_new);
    __syncthreads();
    for (int i = tid; i < n; i += 256) z[i] = expf(z[i] - m_new);
    __syncthreads();
    float ps = 0.f;
    for (int i = 0; i < n; ++i) ps += z[i];
    s_run = s_run * scale_old + ps;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int k = tid + 256 * j;
      if (k < d) {
        float t = acc[j] * scale_old;
        for (int i = 0; i < n; ++i) t = fmaf(z[i], Elem<T>::load(phi + static_cast<long long>(p0 + i) * d + k), t);
        acc[j] = t;
      }
    }
    m_run = m_new;
    __syncthreads();
  }
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int k = tid + 256 * j;
    if (k < d) out[2 + k] = acc[j];
  }
  if (tid == 0) {
    out[0] = m_run;
    out[1] = s_run;
  }
}

// Per request: merge the kSlots slice states and write g = acc / s.
__global__ void __launch_bounds__(256) pool_finish_static_kernel(const __grid_constant__ StaticPoolArgs a,
                                                                 const float* __restrict__ scratch,
                                                                 float* __restrict__ g) {
  const int r = blockIdx.x, d = a.d;
  const float* st = scratch + static_cast<long long>(r) * kSlots * (d + 2);
  float M = -INFINITY;
  for (int c = 0; c < kSlots; ++c) M = fmaxf(M, st[c * (d + 2)]);
  float S = 0.f;
  for (int c = 0; c < kSlots; ++c) {
    const float* sc = st + c * (d + 2);
    if (sc[1] > 0.f) S += sc[1] * expf(sc[0] - M);
  }
  for (int k = threadIdx.x; k < d; k += blockDim.x) {
    float acc = 0.f;
    for (int c = 0; c < kSlots; ++c) {
      const float* sc = st + c * (d + 2);
      if (sc[1] > 0.f) acc = fmaf(sc[2 + k], expf(sc[0] - M), acc);
    }
    g[static_cast<long long>(r) * d + k] = acc / S;
  }
}

// Device address of the static scratch in the current device's context,
// looked up on every call with that device current.  In host code
// `g_anchor_scratch` names only a host-side stand-in, never the device memory,
// so kernels get this address instead.  The lookup allocates nothing; doing it
// per call (instead of caching it per device index) keeps the address right
// after the context has been torn down and created again.
cudaError_t scratch_on_current_device(float** ptr) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_anchor_scratch);
  if (e != cudaSuccess) return e;
  *ptr = static_cast<float*>(p);
  return cudaSuccess;
}

}  // namespace

// Model fields the entry point needs (kept in txs_api.cu).
int model_d(const txs_model* m);
int model_dtype(const txs_model* m);
const float* model_w_pool(const txs_model* m);

}  // namespace txs

using namespace txs;

TXS_API txs_status txs_pool_anchor_static(const txs_model* model, int32_t n_req, const int32_t* beh_offsets,
                                          const void* beh_enc, float* out_g, void* stream) {
  TXS_TRACE();
  if (!model || !beh_offsets || !beh_enc || !out_g || n_req < 1) return TXS_ERR_INVALID_ARG;
  if (beh_offsets[0] != 0) return TXS_ERR_INVALID_ARG;
  for (int r = 0; r < n_req; ++r) {
    if (beh_offsets[r + 1] < beh_offsets[r]) return TXS_ERR_INVALID_ARG;
    if (beh_offsets[r + 1] == beh_offsets[r]) return TXS_ERR_COLD_START;
  }
  const int d = model_d(model);
  if (d > kMaxD) {
    const std::string msg = "txs_pool_anchor_static: d_model " + std::to_string(d) + " is above the limit of " +
                            std::to_string(kMaxD);
    set_last_error(msg.c_str());
    return TXS_ERR_UNSUPPORTED;
  }
  const long long need = static_cast<long long>(n_req) * kSlots * (d + 2);
  if (n_req > kMaxReq || need > kScratchFloats) {
    const std::string msg = "txs_pool_anchor_static: " + std::to_string(n_req) + " requests of width " +
                            std::to_string(d) + " need " + std::to_string(need) +
                            " floats of static scratch; the limit is " + std::to_string(kScratchFloats) +
                            " floats and " + std::to_string(kMaxReq) + " requests";
    set_last_error(msg.c_str());
    return TXS_ERR_UNSUPPORTED;
  }
  float* scratch = nullptr;
  cudaError_t err = scratch_on_current_device(&scratch);
  if (err != cudaSuccess) {
    set_last_error(cudaGetErrorString(err));
    return TXS_ERR_CUDA;
  }
  StaticPoolArgs a;
  a.n_req = n_req;
  a.d = d;
  a.inv_sqrt_d = 1.0f / sqrtf(static_cast<float>(d));
  for (int r = 0; r <= n_req; ++r) a.off[r] = beh_offsets[r];
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (model_dtype(model) == TXS_BF16)
    pool_slices_static_kernel<__nv_bfloat16><<<dim3(kSlots, n_req), 256, 0, s>>>(
        a, static_cast<const __nv_bfloat16*>(beh_enc), model_w_pool(model), scratch);
  else
    pool_slices_static_kernel<float><<<dim3(kSlots, n_req), 256, 0, s>>>(a, static_cast<const float*>(beh_enc),
                                                                         model_w_pool(model), scratch);
  err = cudaGetLastError();
  if (err == cudaSuccess) {
    pool_finish_static_kernel<<<n_req, 256, 0, s>>>(a, scratch, out_g);
    err = cudaGetLastError();
  }
  if (err != cudaSuccess) {
    set_last_error(cudaGetErrorString(err));
    return TXS_ERR_CUDA;
  }
  return TXS_OK;
}
