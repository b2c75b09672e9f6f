// Internal declarations shared by the libtxs translation units (not installed).
#pragma once

#include <cuda.h>
#include <nvtx3/nvToolsExt.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/txs.h"

#define TXS_API extern "C" __attribute__((visibility("default")))

namespace txs {

// NVTX range around a public call (named after the function): it shows in a
// profiler's timeline; without a tool attached it costs a pointer check.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};
#define TXS_TRACE() ::txs::NvtxRange txs_trace_range_(__func__)


// Device-side bounded waits give up after this many SM clock cycles (~1 s at
// 2 GHz), latch TXS_ERR_DEVICE_TIMEOUT and let the kernel wind down.
constexpr long long kSpinCycles = 2000000000LL;

// Kernel classes for the event profiler (txs_profile_*).
enum KernelClass : int {
  KC_PACK = 0, KC_GEMM_QKV, KC_ATTN_SERVING, KC_GEMM_OPROJ, KC_GEMM_Q, KC_ATTN_CROSS,
  KC_GEMM_FFN1, KC_GEMM_FFN2, KC_GEMM_KV, KC_POOL, KC_GLOBAL_KV, KC_RANK, KC_MISC,
  KC_ROW_LN, KC_CAND_MLP, KC_ENC_EMBED, KC_ENC_GEMM, KC_ENC_ATTN, KC_HEAD_DW, KC_GEMM_Q_ATTN, KC_COUNT_
};
static_assert(KC_COUNT_ <= TXS_N_KERNEL_CLASSES, "profiler classes");

// ------------------------------------------------------------------ device helpers

// Programmatic dependent launch: every hot-path kernel lets its successor
// launch early (its prologue then overlaps this kernel's tail) and waits for
// its predecessor's completion before touching global memory.
__device__ __forceinline__ void pdl_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ void latch_status(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

template <typename T> struct Elem;
template <> struct Elem<float> {
  static __device__ __forceinline__ float load(const float* p) { return *p; }
  static __device__ __forceinline__ void store(float* p, float v) { *p = v; }
};
template <> struct Elem<__nv_bfloat16> {
  static __device__ __forceinline__ float load(const __nv_bfloat16* p) { return __bfloat162float(*p); }
  static __device__ __forceinline__ void store(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }
};

// 16-byte vectors of T converted to/from float.
template <typename T> struct Vec16;
template <> struct Vec16<float> {
  static constexpr int N = 4;
  static __device__ __forceinline__ void load(const float* p, float* v) {
    float4 a = *reinterpret_cast<const float4*>(p);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  }
  static __device__ __forceinline__ void store(float* p, const float* v) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  }
};
template <> struct Vec16<__nv_bfloat16> {
  static constexpr int N = 8;
  static __device__ __forceinline__ void load(const __nv_bfloat16* p, float* v) {
    uint4 a = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&a);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float2 f = __bfloat1622float2(h[i]);
      v[2 * i] = f.x; v[2 * i + 1] = f.y;
    }
  }
  static __device__ __forceinline__ void store(__nv_bfloat16* p, const float* v) {
    uint4 a;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&a);
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
    *reinterpret_cast<uint4*>(p) = a;
  }
};

__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}

// max(a, b, c) in one instruction (three-source max.f32, sm_100 and later).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}
// Lane-wise a * b + c and a + b on a pair of fp32 values in one instruction
// (f32x2 arithmetic, sm_100 and later); each lane rounds like fmaf / fadd.
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  uint64_t r;
  asm("{\n\t.reg .b64 x, y, z;\n\t"
      "mov.b64 x, {%1, %2};\n\tmov.b64 y, {%3, %4};\n\tmov.b64 z, {%5, %6};\n\t"
      "fma.rn.f32x2 %0, x, y, z;\n\t}"
      : "=l"(r) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  float2 o;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(o.x), "=f"(o.y) : "l"(r));
  return o;
}
__device__ __forceinline__ float2 fmul2(float2 a, float2 b) {
  uint64_t r;
  asm("{\n\t.reg .b64 x, y;\n\t"
      "mov.b64 x, {%1, %2};\n\tmov.b64 y, {%3, %4};\n\t"
      "mul.rn.f32x2 %0, x, y;\n\t}"
      : "=l"(r) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  float2 o;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(o.x), "=f"(o.y) : "l"(r));
  return o;
}
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  uint64_t r;
  asm("{\n\t.reg .b64 x, y;\n\t"
      "mov.b64 x, {%1, %2};\n\tmov.b64 y, {%3, %4};\n\t"
      "add.rn.f32x2 %0, x, y;\n\t}"
      : "=l"(r) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  float2 o;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(o.x), "=f"(o.y) : "l"(r));
  return o;
}

// Hardware approximations (PTX): reciprocal and 2^x, subnormal results
// flushed to zero.
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ float ex2_approx(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// gelu_erf (above the f32x2 helpers) with erf from the rational approximation
// of Abramowitz & Stegun, Handbook of Mathematical Functions (1964), formula
// 7.1.26: for z >= 0, 1 - erf(z) = t P(t) exp(-z^2) with t = 1 / (1 + p z),
// P(t) = a1 + t (a2 + t (a3 + t (a4 + t a5))), absolute error at most 1.5e-7.
// Since erf is odd, with a = |x| and z = a / sqrt 2 both signs reduce to
//   GELU(x) = 0.5 x (1 + erf(x / sqrt 2)) = max(x, 0) - 0.5 a t P(t) exp(-a^2 / 2),
// which needs no sign handling and never forms 1 - (1 - small).  The bf16
// tensor-core epilogues use it on two values at once (f32x2 multiplies and
// multiply-adds; the 0.5 and 1 / sqrt 2 are folded into the constants), with
// the hardware reciprocal and 2^x; in fp32 the result stays within a few
// 1e-7 of 0.5 |x| of the exact GELU, against bf16 outputs with a relative
// step of 2^-8.
__device__ __forceinline__ float2 gelu_erf_as2(float2 x) {
  const float2 a = make_float2(fabsf(x.x), fabsf(x.y));
  constexpr float kP = 0.3275911f * 0.70710678118654752f;        // p / sqrt 2
  const float2 den = ffma2(a, make_float2(kP, kP), make_float2(1.0f, 1.0f));
  const float2 t = make_float2(rcp_approx(den.x), rcp_approx(den.y));
  // 0.5 P(t)
  float2 q = ffma2(t, make_float2(0.5f * 1.061405429f, 0.5f * 1.061405429f),
                   make_float2(0.5f * -1.453152027f, 0.5f * -1.453152027f));
  q = ffma2(t, q, make_float2(0.5f * 1.421413741f, 0.5f * 1.421413741f));
  q = ffma2(t, q, make_float2(0.5f * -0.284496736f, 0.5f * -0.284496736f));
  q = ffma2(t, q, make_float2(0.5f * 0.254829592f, 0.5f * 0.254829592f));
  // exp(-a^2 / 2) = 2^(-a^2 log2(e) / 2)
  constexpr float kE = -0.5f * 1.4426950408889634f;
  const float2 zz = fmul2(a, fmul2(a, make_float2(kE, kE)));
  const float2 e = make_float2(ex2_approx(zz.x), ex2_approx(zz.y));
  const float2 g = fmul2(fmul2(fmul2(a, t), q), e);
  return fadd2(make_float2(fmaxf(x.x, 0.0f), fmaxf(x.y, 0.0f)), make_float2(-g.x, -g.y));
}

// Index of the segment that contains `row` in an exclusive-offset array
// off[0..n] (off[0] == 0, non-decreasing): largest r with off[r] <= row.
__device__ __forceinline__ int find_segment(const int* off, int n, int row) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (__ldg(off + mid) <= row) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// ------------------------------------------------------------------ host side

// Launch with programmatic stream serialization (see pdl_wait).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

struct Prof;  // event profiler (txs_api.cu)
void prof_begin(int cls, cudaStream_t s);
void prof_end(int cls, cudaStream_t s);

// Epilogue kinds shared by the SIMT and tensor-core GEMMs.
enum Epi : int {
  EPI_BIAS = 0,       // out = acc + bias
  EPI_BIAS_GELU = 1,  // out = GELU(acc + bias)
  EPI_KV = 2,         // out = acc + bias, rows remapped into the cache, cols into [l][K|V]
  EPI_LN = 3,         // out = LN(acc + bias + res) over the full row (N == d)
  EPI_LN_HEAD = 4,    // z = LN(...); logits = z Weff_z + xlog; probs = softmax(logits)
  EPI_ATTN_LG = 5,    // q = acc + bias; out = LOCAL_GLOBAL cross-attention of q (tensor cores, bf16)
  EPI_SERVE = 6,      // q, k, v = acc + bias of one head; out = serving-stream attention (tensor cores, bf16)
};

// Arguments of every GEMM epilogue; unused fields are ignored.
struct EpiArgs {
  int epi;
  int M, N, K;
  const float* bias;      // [N]
  void* out;              // row-major, leading dimension ldo (elements)
  long long ldo;
  const void* res;        // residual, leading dimension ldr (EPI_LN*)
  long long ldr;
  const float* gamma;     // LN gain/bias [N]
  const float* beta;
  float ln_eps;
  // EPI_KV: row remap (request of row from seg_off[0..n_seg]; out row =
  // dst_row0[r] + row - seg_off[r]) and column blocks of width col_blk placed
  // col_blk_stride elements apart.
  const int* seg_off;
  const int* dst_row0;
  int n_seg;
  int col_blk;
  long long col_blk_stride;
  // EPI_LN_HEAD
  const float* weff_z;    // [N, n_act]  (W_dec[:d] Q_dec^T)
  const float* xlog;      // [n_cand_rows, n_act] (x W_dec[d:] Q_dec^T + b_dec Q_dec^T)
  int n_act;
  int n_cand_rows;        // rows >= this are context rows (no head output)
  float* logits;
  float* probs;
  int* status;
  // EPI_KV on the tensor cores: when kv_host_up is set (host [in_off (R+1) |
  // dst0 (R)] and kv_host_len [R]) and n_seg fits the kernel's parameter
  // block, the launch carries these values by value; the kernel uses them for
  // its row remap and writes them to kv_dev_up / kv_dev_len (seg_off and the
  // lengths the later kernels read), so no separate upload is needed.
  const int* kv_host_up;
  const int* kv_host_len;
  int* kv_dev_up;
  int* kv_dev_len;
  // EPI_ATTN_LG: the accumulator row is a query q = acc + bias of packed row
  // `row` (request att_row_req[row]); the epilogue writes, per head, the
  // softmax-weighted values of that request's last att_l_local cached rows
  // (att_k / att_v: the layer's cache, [cap_total][att_dkv] bf16, request r
  // at row att_kv_off[r], att_kv_len[r] rows) and of its anchor
  // (att_kg / att_vg [R][att_dkv] fp32); query head h reads K/V head
  // h / att_group.
  const void* att_k;
  const void* att_v;
  const float* att_kg;
  const float* att_vg;
  const int* att_row_req;
  const int* att_kv_off;
  const int* att_kv_len;
  int att_dkv, att_group, att_dh, att_l_local;
  float att_scale_log2;   // log2(e) / sqrt(d_h)
  // rows at or past att_n_cand (the context tokens, several requests per
  // warp) are not attended here: their q (bf16) goes to att_q_ctx at the
  // same row and column, for a separate launch over those rows
  int att_n_cand;
  void* att_q_ctx;
  // EPI_SERVE: tile n holds q, k, v (d_h columns each, the weights' output
  // columns permuted per head) of head n for candidate row `row` (request
  // srv_row_req[row]); the epilogue writes that head's serving-stream
  // attention output (App. B mask: the request's srv_S context rows and the
  // row itself) to out[row][n d_h ...].  The context rows' k and v are rows
  // r srv_S + t of srv_ctx ([R S][3 srv_d] bf16, columns [q | k | v]).
  const void* srv_ctx;
  const int* srv_row_req;
  int srv_S, srv_d;
  float srv_scale_log2;   // log2(e) / sqrt(d_h)
};
// Largest request count whose offsets an EPI_KV launch carries by value.
constexpr int kKvParamReq = 1000;

// Launchers (return cudaError_t of the launch).
// fp32 A; B float or bf16; fp32 output (EPI_KV with seg_off == nullptr keeps rows)
template <typename TB>
cudaError_t launch_gemm_simt(const float* A, long long lda, const TB* B, const EpiArgs& e,
                             float* tmp, cudaStream_t s, int cls);
// GELU of the GEMM epilogues on device float arrays (variant 0: bf16
// tensor-core epilogue, 1: fp32 path), for tests.
cudaError_t launch_gelu_eval(const float* x, float* y, long long n, int variant, cudaStream_t s);
// One bounded wait that runs out (about a second), latching TXS_ERR_DEVICE_TIMEOUT.
cudaError_t launch_wait_timeout_probe(int* status, cudaStream_t s);
cudaError_t launch_gemm_tc(const __nv_bfloat16* A, long long lda, const __nv_bfloat16* B,
                           const EpiArgs& e, cudaStream_t s, int cls);
bool tc_gemm_supported(int N, int K, int epi);
namespace tc {
int num_sms();   // streaming multiprocessors of the current device
}

template <typename T>
cudaError_t launch_serving_attn(const T* qkv, T* out, const int* row_req, int n_rows, int n_cand_rows, int S, int H,
                                int d, cudaStream_t s);
// LOCAL_GLOBAL cross-attention with the window in shared memory; cudaErrorNotSupported
// when the window is longer than 16 rows or d_h is not 32 / 64.
template <typename T>
cudaError_t launch_cross_attn_lg(const T* q, T* out, const T* Kc, const T* Vc, const int* cand_off_dev,
                                 const int* cand_off_host, int n_req, int n_cand, int S, const int* kv_off,
                                 const int* kv_len, const float* Kg, const float* Vg, int l_local, int H, int Hkv,
                                 int d, cudaStream_t s);
// LOCAL_GLOBAL cross-attention of the context-token rows only (rows n_cand +
// r S + j), one warp per (row, head), for the fused query projection that
// leaves those rows' q in `q` (row stride d).
cudaError_t launch_ctx_attn_lg(const __nv_bfloat16* q, __nv_bfloat16* out, const __nv_bfloat16* Kc,
                               const __nv_bfloat16* Vc, int n_req, int n_cand, int S, const int* kv_off,
                               const int* kv_len, const float* Kg, const float* Vg, int l_local, int H, int Hkv,
                               int d, cudaStream_t s);
template <typename T>
cudaError_t launch_cross_attn(const T* q, T* out, const T* Kc, const T* Vc, const int* row_req, int n_rows,
                              const int* kv_off, const int* kv_len, const float* Kg, const float* Vg, int l_local,
                              int mode, int H, int Hkv, int d, cudaStream_t s);

// FULL-mode cross-attention on the tensor cores (bf16): one CTA per
// (128-query tile, request, head).
bool fa_full_supported(int d, int H, long long cap_total);
cudaError_t launch_fa_full(const __nv_bfloat16* q, __nv_bfloat16* out, const __nv_bfloat16* Kc,
                           const __nv_bfloat16* Vc, long long cap_total, const int* cand_off_dev,
                           const int* cand_off_host, const int* kv_off, const int* kv_len, int n_req, int n_cand,
                           int S, int H, int Hkv, int d, int* status, cudaStream_t s);

extern const int kPoolChunk;
template <typename T>
cudaError_t launch_pool(const T* phi, const int* seg_off, int R, int max_rows, const float* w_pool, int d,
                        int max_chunks, float* part, int merge_existing, float* st_m, float* st_s, float* st_acc,
                        float* g, int* counter, int* status, cudaStream_t s);
// Per-event anchors of one user's stream: g[t] = attention pooling of
// phi[0 .. ends[t]); also writes ev_off[t] = off_user, ev_len[t] = ends[t]
// (ends: host, at most 4096 events; d <= 512).  `part`: scratch of
// prefix_pool_scratch_floats(max end, d) floats.
size_t prefix_pool_scratch_floats(int max_end, int d);
template <typename T>
cudaError_t launch_prefix_pool(const T* phi, const int* ends, int n_ev, int off_user, const float* w_pool, int d,
                               float* part, float* g, int* ev_off, int* ev_len, cudaStream_t s);
template <typename T>
cudaError_t launch_anchor_proj(const float* g, const T* Wt_kv, const float* b_kv, float* gkv, int R, int d, int dkv,
                               int n_layers, cudaStream_t s);
template <typename T>
cudaError_t launch_transpose(const T* W, T* Wt, int rows, int cols, cudaStream_t s);
template <typename T>
cudaError_t launch_to_f32(const T* src, float* dst, long long n, cudaStream_t s);
template <typename T>
cudaError_t launch_fold_dw(const T* W_w, const T* b_w, const T* W_d2, const T* b_d2, const T* Q_dec, float* weff_x,
                           float* cdec, float* w2q, int d, int dw_in, int dw_out, int Fh, int k, cudaStream_t s);
template <typename T>
cudaError_t launch_dw_gather(const T* Z, const T* cand, T* Z2, int n_cand, int d, int dw_in, cudaStream_t s);
template <typename T>
cudaError_t launch_dw_head(const T* Hd, int Fh, const float* w2q, const float* xlog, int na, int n_cand,
                           float* logits, float* probs, cudaStream_t s);
template <typename T>
cudaError_t launch_fold_head(const T* W_dec, const T* b_dec, const T* Q_dec, float* weff, float* cdec, int d, int k,
                             cudaStream_t s);
cudaError_t launch_hash(const void* p, long long bytes, uint64_t salt, unsigned long long* out, cudaStream_t s);

extern const int kMaxReqParam;
// dst_a[0..n_a) = src_a, dst_b[0..n_b) = src_b (host arrays) by one kernel
// whose parameters carry the values; cudaErrorNotSupported above
// kUploadParamInts ints in all (the caller then copies through pinned memory).
extern const int kUploadParamInts;
cudaError_t launch_upload_ints(int* dst_a, const int* src_a, int n_a, int* dst_b, const int* src_b, int n_b,
                               cudaStream_t s);
template <typename T>
cudaError_t launch_pack(int n_req, const int* cand_off_host, int S, int d, int na, const T* cand, const T* ctx, T* X,
                        int* row_req, int* cand_off_dev, const float* weff_x, const float* cdec, float* xlog,
                        cudaStream_t s);
cudaError_t launch_rank(int n_req, const int* cand_off_host, const float* probs, int na, int action, int top_k,
                        int* out, cudaStream_t s);

// Behavior-stream encoder (k_encoder.cu).  Query rows per attention CTA for
// calls whose users have at most `max_new_rows` new rows each.
int enc_query_tile(int max_new_rows);
template <typename T>
cudaError_t launch_enc_embed(const T* subj, const int* types, const T* E_type, T* X, long long n, int d, int dt,
                             int n_types, int* status, cudaStream_t s);
template <typename T>
cudaError_t launch_enc_rel_prep(const T* beta, float* out, int n, cudaStream_t s);
template <typename T>
cudaError_t launch_enc_attn(const T* q, const T* K, const T* V, T* out, const int* in_off, const int* dst0,
                            const int* slot_off, const int* tile_off, int n_req, int n_tiles, int query_tile,
                            const float* beta_log2, int n_rel, int window, int H, int d, int* status,
                            cudaStream_t s);
// The same on the tensor cores (bf16; 128-row query tiles, 128-key tiles
// aligned on each user's position axis); cudaErrorNotSupported unless d_h is
// 32 or 64 and n_rel <= 8192.
bool enc_attn_tc_supported(int d, int H, int n_rel);
cudaError_t launch_enc_attn_tc(const __nv_bfloat16* q, const __nv_bfloat16* K, const __nv_bfloat16* V,
                               __nv_bfloat16* out, long long cap_total, const int* in_off, const int* dst0,
                               const int* slot_off, const int* tile_off, int n_req, int n_tiles,
                               const float* beta_log2, int n_rel, int window, int H, int d, int* status,
                               cudaStream_t s);
void set_last_error(const char* msg);

}  // namespace txs
