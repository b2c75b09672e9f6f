// fp32 instantiation of the dense projections (CUDA cores, fp32 FMA).
//
// The fp32 model dtype keeps every operand in fp32 (no reduced-precision tensor
// math), so its GEMMs run here: C = A B^T with A [M, K], B [N, K] row-major,
// followed by the same epilogue kinds as the tensor-core path.  Row-wise
// LayerNorm epilogues (Sec. 4.1.2 crossAttend equation) need the whole row, so
// for them the GEMM writes acc + bias + residual to a scratch matrix and
// row_ln_kernel normalises it (and, for the last layer, applies the action head
// of Sec. 4.1.3).
#include "txs_internal.cuh"

namespace txs {

namespace {

constexpr int TM = 64, TN = 64, TK = 16;

template <int EPI, typename TB>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const float* __restrict__ A, long long lda,
                                                        const TB* __restrict__ B, const EpiArgs e,
                                                        float* __restrict__ tmp) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ float As[TK][TM + 4];
  __shared__ float Bs[TK][TN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int m0 = blockIdx.x * TM, n0 = blockIdx.y * TN;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int k0 = 0; k0 < e.K; k0 += TK) {
    for (int i = threadIdx.x; i < TM * TK; i += 256) {
      const int mm = i / TK, kk = i % TK;
      const int gm = m0 + mm, gk = k0 + kk;
      As[kk][mm] = (gm < e.M && gk < e.K) ? A[static_cast<long long>(gm) * lda + gk] : 0.f;
      const int gn = n0 + mm;
      Bs[kk][mm] = (gn < e.N && gk < e.K) ? Elem<TB>::load(B + static_cast<long long>(gn) * e.K + gk) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }

#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= e.M) continue;
    long long orow = m;
    if constexpr (EPI == EPI_KV) {
      if (e.seg_off) {   // rows remapped into cache slots; identity otherwise
        const int r = find_segment(e.seg_off, e.n_seg, m);
        orow = static_cast<long long>(e.dst_row0[r]) + (m - e.seg_off[r]);
      }
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= e.N) continue;
      float v = acc[i][j] + e.bias[n];
      if constexpr (EPI == EPI_BIAS) {
        static_cast<float*>(e.out)[orow * e.ldo + n] = v;
      } else if constexpr (EPI == EPI_BIAS_GELU) {
        static_cast<float*>(e.out)[orow * e.ldo + n] = gelu_erf(v);
      } else if constexpr (EPI == EPI_KV) {
        const int blk = n / e.col_blk;
        static_cast<float*>(e.out)[static_cast<long long>(blk) * e.col_blk_stride + orow * e.ldo +
                                   (n - blk * e.col_blk)] = v;
      } else {
        v += static_cast<const float*>(e.res)[static_cast<long long>(m) * e.ldr + n];
        tmp[static_cast<long long>(m) * e.N + n] = v;
      }
    }
  }
}

// One warp per row: LayerNorm of tmp[row, 0:N] (two-pass mean / biased
// variance), then either store (EPI_LN) or the action head (EPI_LN_HEAD).
template <int EPI>
__global__ void __launch_bounds__(256) row_ln_kernel(const float* __restrict__ tmp, const EpiArgs e) {
  pdl_launch_dependents();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * 8 + warp;
  if (row >= e.M) return;
  const int N = e.N;
  const float* x = tmp + static_cast<long long>(row) * N;
  float v[32];
  float sum = 0.f;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const int c = lane + 32 * i;
    v[i] = c < N ? x[c] : 0.f;
    sum += v[i];
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  const float mean = sum / N;
  float sq = 0.f;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const int c = lane + 32 * i;
    if (c < N) sq += (v[i] - mean) * (v[i] - mean);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
  const float rstd = rsqrtf(sq / N + e.ln_eps);
  float lg[16];
#pragma unroll
  for (int a = 0; a < 16; ++a) lg[a] = 0.f;
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    const int c = lane + 32 * i;
    if (c >= N) continue;
    const float y = (v[i] - mean) * rstd * e.gamma[c] + e.beta[c];
    if constexpr (EPI == EPI_LN) {
      static_cast<float*>(e.out)[static_cast<long long>(row) * e.ldo + c] = y;
    } else {
#pragma unroll
      for (int a = 0; a < 16; ++a)
        if (a < e.n_act) lg[a] = fmaf(y, e.weff_z[static_cast<long long>(c) * e.n_act + a], lg[a]);
    }
  }
  if constexpr (EPI == EPI_LN_HEAD) {
    if (row >= e.n_cand_rows) return;
#pragma unroll
    for (int a = 0; a < 16; ++a)
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) lg[a] += __shfl_xor_sync(0xffffffffu, lg[a], o);
    if (lane == 0) {
      const int na = e.n_act;
      float mx = -INFINITY;
      for (int a = 0; a < na; ++a) {
        lg[a] += e.xlog[static_cast<long long>(row) * na + a];
        mx = fmaxf(mx, lg[a]);
      }
      float s = 0.f;
      float p[16];
      for (int a = 0; a < na; ++a) {
        p[a] = expf(lg[a] - mx);
        s += p[a];
      }
      for (int a = 0; a < na; ++a) {
        e.logits[static_cast<long long>(row) * na + a] = lg[a];
        if (e.probs) e.probs[static_cast<long long>(row) * na + a] = p[a] / s;
      }
    }
  }
}

}  // namespace

template <typename TB>
cudaError_t launch_gemm_simt(const float* A, long long lda, const TB* B, const EpiArgs& e, float* tmp,
                             cudaStream_t s, int cls) {
  if (e.M == 0) return cudaSuccess;
  if ((e.epi == EPI_LN || e.epi == EPI_LN_HEAD) && e.N > 1024) return cudaErrorInvalidValue;
  dim3 grid((e.M + TM - 1) / TM, (e.N + TN - 1) / TN);
  cudaError_t err0 = cudaSuccess;
  prof_begin(cls, s);
  switch (e.epi) {
    case EPI_BIAS: err0 = launch_pdl(gemm_simt_kernel<EPI_BIAS, TB>, grid, dim3(256), 0, s, A, lda, B, e, tmp); break;
    case EPI_BIAS_GELU: err0 = launch_pdl(gemm_simt_kernel<EPI_BIAS_GELU, TB>, grid, dim3(256), 0, s, A, lda, B, e, tmp); break;
    case EPI_KV: err0 = launch_pdl(gemm_simt_kernel<EPI_KV, TB>, grid, dim3(256), 0, s, A, lda, B, e, tmp); break;
    case EPI_LN:
    case EPI_LN_HEAD:
      err0 = launch_pdl(gemm_simt_kernel<EPI_LN, TB>, grid, dim3(256), 0, s, A, lda, B, e, tmp);
      break;
    default: return cudaErrorInvalidValue;
  }
  cudaError_t err = err0 != cudaSuccess ? err0 : cudaGetLastError();
  prof_end(cls, s);
  if (err != cudaSuccess) return err;
  if (e.epi == EPI_LN || e.epi == EPI_LN_HEAD) {
    prof_begin(KC_ROW_LN, s);
    const int blocks = (e.M + 7) / 8;
    if (e.epi == EPI_LN) err = launch_pdl(row_ln_kernel<EPI_LN>, dim3(blocks), dim3(256), 0, s, tmp, e);
    else err = launch_pdl(row_ln_kernel<EPI_LN_HEAD>, dim3(blocks), dim3(256), 0, s, tmp, e);
    prof_end(KC_ROW_LN, s);
  }
  return err;
}

template cudaError_t launch_gemm_simt<float>(const float*, long long, const float*, const EpiArgs&, float*,
                                             cudaStream_t, int);
template cudaError_t launch_gemm_simt<__nv_bfloat16>(const float*, long long, const __nv_bfloat16*, const EpiArgs&,
                                                     float*, cudaStream_t, int);

}  // namespace txs
