// Kernels of the behavior-stream encoder Phi_behavior (Sec. 4.1.1) and its
// incremental update (App. D, incremental-encoding remark):
//   * enc_embed_kernel: behavior token = [subject row, E_type[type]];
//   * enc_rel_prep_kernel: the per-head relative-bias tables in fp32, scaled
//     by log2(e) for the exp2 softmax;
//   * enc_attn_kernel: causal self-attention with the relative position bias
//     beta_h[min(i - j, R - 1)], for a set of new rows of each user against
//     that user's cached keys/values of the same layer (the new rows' own
//     keys/values are already in the cache when it runs).
// The dense projections of the encoder layer run on the library's GEMMs.
#include <algorithm>
#include <cmath>

#include "txs_internal.cuh"

namespace txs {
namespace {

constexpr int kEncKeys = 32;     // keys per tile: one per lane
constexpr int kEncThreads = 256; // 8 warps

template <typename T>
__global__ void __launch_bounds__(256)
    enc_embed_kernel(const T* __restrict__ subj, const int* __restrict__ types, const T* __restrict__ E_type,
                     T* __restrict__ X, long long n, int d, int dt, int n_types, int* status) {
  pdl_wait();
  pdl_launch_dependents();
  const int ds = d - dt;
  const long long total = n * d;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long row = i / d;
    const int c = static_cast<int>(i - row * d);
    T v;
    if (c < ds) {
      v = subj[row * ds + c];
    } else {
      const int t = types[row];
      if (t < 0 || t >= n_types) {
        latch_status(status, TXS_ERR_BOUNDS);
        Elem<T>::store(&v, 0.f);
      } else {
        v = E_type[static_cast<long long>(t) * dt + (c - ds)];
      }
    }
    X[i] = v;
  }
}

template <typename T>
__global__ void enc_rel_prep_kernel(const T* __restrict__ beta, float* __restrict__ out, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) out[i] = Elem<T>::load(beta + i) * 1.4426950408889634f;
}

struct EncAttnArgs {
  const void* q;        // [n][d] queries of the new rows (model dtype)
  const void* K;        // [cap_total][d] keys of this layer, by cache slot
  const void* V;        // [cap_total][d] values
  void* out;            // [n][d]
  const int* in_off;    // [R+1] new rows of user r: in_off[r] .. in_off[r+1]
  const int* dst0;      // [R]   slot of user r's first new row
  const int* slot_off;  // [R+1] slots of user r: slot_off[r] .. slot_off[r+1]
  const int* tile_off;  // [R+1] query tiles of user r: tile_off[r] .. tile_off[r+1]
  const float* beta;    // [H][n_rel] relative bias times log2(e)
  int n_req, n_rel, window, d;
  float scale_log2;     // log2(e) / sqrt(d_h)
  int* status;
};

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One CTA per (query tile of one user, head).  Each warp owns RPW query rows;
// key tiles of 32 positions, aligned to multiples of 32 of the user's
// position axis, are staged in shared memory (next tile prefetched into
// registers).  A row's arithmetic depends only on its own position and the
// keys, never on which other rows share the CTA: fully masked tiles leave its
// state untouched.  So encoding tokens incrementally gives bit-identical rows
// to encoding the stream at once.
template <typename T, int DH, int RPW>
__global__ void __launch_bounds__(kEncThreads) enc_attn_kernel(const EncAttnArgs a) {
  constexpr int NW = kEncThreads / 32, QT = NW * RPW, NV = DH / 32;
  constexpr int VN = Vec16<T>::N;                 // elements per 16-byte vector
  constexpr int VROW = DH / VN;                   // vectors per key row
  constexpr int VTILE = kEncKeys * VROW;          // vectors per K (or V) tile
  constexpr int VPT = (VTILE + kEncThreads - 1) / kEncThreads;
  __shared__ float sQ[QT][DH];
  __shared__ float sK[kEncKeys][DH + 1];
  __shared__ float sV[kEncKeys][DH];

  pdl_wait();
  pdl_launch_dependents();
  const int h = blockIdx.y;
  const int r = find_segment(a.tile_off, a.n_req, blockIdx.x);
  const int t = blockIdx.x - __ldg(a.tile_off + r);
  const int row0 = __ldg(a.in_off + r) + t * QT;
  const int nrows = min(QT, __ldg(a.in_off + r + 1) - row0);
  const int base = __ldg(a.slot_off + r);
  const int cap = __ldg(a.slot_off + r + 1) - base;
  const int pos0 = __ldg(a.dst0 + r) - base + t * QT;  // position of row0 on the user's axis
  if (nrows <= 0) return;
  if (pos0 < 0 || pos0 + nrows > cap) {
    if (threadIdx.x == 0) latch_status(a.status, TXS_ERR_BOUNDS);
    return;
  }
  const T* q = static_cast<const T*>(a.q);
  const T* K = static_cast<const T*>(a.K);
  const T* V = static_cast<const T*>(a.V);
  const int col = h * DH;
  for (int i = threadIdx.x; i < QT * VROW; i += kEncThreads) {
    const int rr = i / VROW, c = (i % VROW) * VN;
    float v[VN];
    if (rr < nrows) {
      Vec16<T>::load(q + static_cast<long long>(row0 + rr) * a.d + col + c, v);
#pragma unroll
      for (int e = 0; e < VN; ++e) v[e] *= a.scale_log2;
    } else {
#pragma unroll
      for (int e = 0; e < VN; ++e) v[e] = 0.f;
    }
#pragma unroll
    for (int e = 0; e < VN; ++e) sQ[rr][c + e] = v[e];
  }

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float m[RPW], l[RPW], acc[RPW][NV];
#pragma unroll
  for (int i = 0; i < RPW; ++i) {
    m[i] = -INFINITY;
    l[i] = 0.f;
#pragma unroll
    for (int v = 0; v < NV; ++v) acc[i][v] = 0.f;
  }
  const int p_last = pos0 + nrows - 1;
  const int lo = a.window > 0 ? max(0, pos0 - a.window + 1) : 0;
  const int j_begin = lo & ~(kEncKeys - 1);
  const float* beta = a.beta + static_cast<long long>(h) * a.n_rel;

  // register prefetch of one K and V tile (keys beyond p_last read as zero)
  uint4 rk[VPT], rv[VPT];
  auto fetch = [&](int j0) {
#pragma unroll
    for (int u = 0; u < VPT; ++u) {
      const int i = threadIdx.x + u * kEncThreads;
      rk[u] = make_uint4(0, 0, 0, 0);
      rv[u] = make_uint4(0, 0, 0, 0);
      if (i < VTILE) {
        const int kk = i / VROW, c = (i % VROW) * VN;
        const int j = j0 + kk;
        if (j <= p_last) {
          const long long o = static_cast<long long>(base + j) * a.d + col + c;
          rk[u] = __ldg(reinterpret_cast<const uint4*>(K + o));
          rv[u] = __ldg(reinterpret_cast<const uint4*>(V + o));
        }
      }
    }
  };
  auto stash = [&]() {
#pragma unroll
    for (int u = 0; u < VPT; ++u) {
      const int i = threadIdx.x + u * kEncThreads;
      if (i < VTILE) {
        const int kk = i / VROW, c = (i % VROW) * VN;
        float fk[VN], fv[VN];
        Vec16<T>::load(reinterpret_cast<const T*>(&rk[u]), fk);
        Vec16<T>::load(reinterpret_cast<const T*>(&rv[u]), fv);
#pragma unroll
        for (int e = 0; e < VN; ++e) {
          sK[kk][c + e] = fk[e];
          sV[kk][c + e] = fv[e];
        }
      }
    }
  };

  if (j_begin <= p_last) fetch(j_begin);
  for (int j0 = j_begin; j0 <= p_last; j0 += kEncKeys) {
    __syncthreads();  // previous tile consumed; sQ staged (first pass)
    stash();
    __syncthreads();
    if (j0 + kEncKeys <= p_last) fetch(j0 + kEncKeys);
    float kr[DH];
#pragma unroll
    for (int c = 0; c < DH; ++c) kr[c] = sK[lane][c];
    const int j = j0 + lane;
#pragma unroll
    for (int rr = 0; rr < RPW; ++rr) {
      const int qi = warp * RPW + rr;
      if (qi >= nrows) break;  // warp-uniform
      const int dist = pos0 + qi - j;
      const bool vis = dist >= 0 && (a.window <= 0 || dist < a.window);
      float s = -INFINITY;
      if (vis) {
        float dot = 0.f;
#pragma unroll
        for (int c = 0; c < DH; ++c) dot = fmaf(sQ[qi][c], kr[c], dot);
        s = dot + __ldg(beta + min(dist, a.n_rel - 1));
      }
      const float tmax = warp_max(s);
      if (tmax == -INFINITY) continue;  // no visible key in this tile for this row
      const float mn = fmaxf(m[rr], tmax);
      const float corr = exp2f(m[rr] - mn);
      const float pj = vis ? exp2f(s - mn) : 0.f;
      l[rr] = l[rr] * corr + warp_sum(pj);
#pragma unroll
      for (int v = 0; v < NV; ++v) acc[rr][v] *= corr;
#pragma unroll 8
      for (int k = 0; k < kEncKeys; ++k) {
        const float pk = __shfl_sync(0xffffffffu, pj, k);
#pragma unroll
        for (int v = 0; v < NV; ++v) acc[rr][v] = fmaf(pk, sV[k][lane + 32 * v], acc[rr][v]);
      }
      m[rr] = mn;
    }
  }
  T* out = static_cast<T*>(a.out);
#pragma unroll
  for (int rr = 0; rr < RPW; ++rr) {
    const int qi = warp * RPW + rr;
    if (qi >= nrows) break;
    const float inv = 1.f / l[rr];
#pragma unroll
    for (int v = 0; v < NV; ++v)
      Elem<T>::store(out + static_cast<long long>(row0 + qi) * a.d + col + lane + 32 * v, acc[rr][v] * inv);
  }
}

template <typename T, int DH, int RPW>
cudaError_t launch_attn_cfg(const EncAttnArgs& a, int n_tiles, int H, cudaStream_t s) {
  return launch_pdl(enc_attn_kernel<T, DH, RPW>, dim3(n_tiles, H), dim3(kEncThreads), 0, s, a);
}

}  // namespace

int enc_query_tile(int max_new_rows) { return max_new_rows <= 8 ? 8 : 32; }

template <typename T>
cudaError_t launch_enc_embed(const T* subj, const int* types, const T* E_type, T* X, long long n, int d, int dt,
                             int n_types, int* status, cudaStream_t s) {
  if (n == 0) return cudaSuccess;
  const long long total = n * d;
  const int blocks = static_cast<int>(std::min<long long>((total + 255) / 256, 152LL * 16));
  prof_begin(KC_ENC_EMBED, s);
  cudaError_t e = launch_pdl(enc_embed_kernel<T>, dim3(blocks), dim3(256), 0, s, subj, types, E_type, X, n, d, dt,
                             n_types, status);
  prof_end(KC_ENC_EMBED, s);
  return e;
}

template <typename T>
cudaError_t launch_enc_rel_prep(const T* beta, float* out, int n, cudaStream_t s) {
  enc_rel_prep_kernel<T><<<(n + 255) / 256, 256, 0, s>>>(beta, out, n);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_enc_attn(const T* q, const T* K, const T* V, T* out, const int* in_off, const int* dst0,
                            const int* slot_off, const int* tile_off, int n_req, int n_tiles, int query_tile,
                            const float* beta_log2, int n_rel, int window, int H, int d, int* status,
                            cudaStream_t s) {
  if (n_tiles == 0) return cudaSuccess;
  const int dh = d / H;
  EncAttnArgs a;
  a.q = q;
  a.K = K;
  a.V = V;
  a.out = out;
  a.in_off = in_off;
  a.dst0 = dst0;
  a.slot_off = slot_off;
  a.tile_off = tile_off;
  a.beta = beta_log2;
  a.n_req = n_req;
  a.n_rel = n_rel;
  a.window = window;
  a.d = d;
  a.scale_log2 = 1.4426950408889634f / std::sqrt(static_cast<float>(dh));
  a.status = status;
  cudaError_t e = cudaErrorInvalidValue;
  prof_begin(KC_ENC_ATTN, s);
  if (dh == 64 && query_tile == 8) e = launch_attn_cfg<T, 64, 1>(a, n_tiles, H, s);
  else if (dh == 64 && query_tile == 32) e = launch_attn_cfg<T, 64, 4>(a, n_tiles, H, s);
  else if (dh == 32 && query_tile == 8) e = launch_attn_cfg<T, 32, 1>(a, n_tiles, H, s);
  else if (dh == 32 && query_tile == 32) e = launch_attn_cfg<T, 32, 4>(a, n_tiles, H, s);
  prof_end(KC_ENC_ATTN, s);
  return e;
}

#define TXS_INST(T)                                                                                               \
  template cudaError_t launch_enc_embed<T>(const T*, const int*, const T*, T*, long long, int, int, int, int*,    \
                                           cudaStream_t);                                                         \
  template cudaError_t launch_enc_rel_prep<T>(const T*, float*, int, cudaStream_t);                               \
  template cudaError_t launch_enc_attn<T>(const T*, const T*, const T*, T*, const int*, const int*, const int*,  \
                                          const int*, int, int, int, const float*, int, int, int, int, int*,      \
                                          cudaStream_t);
TXS_INST(float)
TXS_INST(__nv_bfloat16)
#undef TXS_INST

}  // namespace txs
