// Projections followed by residual + LayerNorm (and, for the last layer, the
// action head), with the row split across a thread-block cluster.
//
// Out = LN(A W + b + residual) needs whole rows (Sec. 4.1.2 crossAttend
// equation, post-LN).  A 128 x d tile computed by one CTA leaves most SMs idle
// when there are few rows, so here a cluster of CS = d / 128 CTAs shares each
// 128-row tile: CTA k computes columns [128 k, 128 k + 128) (tcgen05, TMEM
// double buffer, persistent over the cluster's row tiles) and the row
// statistics are combined across the cluster through distributed shared
// memory: every epilogue warp publishes the mean and the sum of squared
// deviations of its 128 columns to all CTAs of the cluster, and each row
// merges the CS partial results (pairwise-update formula for equal counts).
// The CTAs of a cluster read the same activation rows: each loads 1 / CS of
// every activation stage and multicasts it into the stage of all CTAs (a stage
// is reloaded once every CTA's MMAs have released it).  The epilogue warps
// form two groups that take alternate tiles (group g the tiles of TMEM buffer
// g) when each cluster has several row tiles, so one tile's normalisation
// runs while the other group waits for its cluster's statistics.  With the head, each CTA's
// partial logits z . W_eff_z go to rank 0, which adds the x part, applies the
// softmax and writes logits and probabilities (Sec. 4.1.3 action-decoding
// equation).
#include "tc_ptx.cuh"

namespace txs {
namespace tcln {

using namespace tc;

constexpr int BN = 128;                 // columns per CTA
constexpr int kWarps = 8;               // epilogue warps: two groups of one per TMEM lane quarter
constexpr int kGroupWarps = kWarps / 2;
constexpr int NUM_THREADS = 64 + 32 * kWarps;

template <int CS, bool HEAD, bool PING>
struct LnShape {
  static constexpr int NAP = 4;                                    // head actions padded to 4
  static constexpr int P = PING ? CS : 2 * CS;                     // partials per row (per CTA or half)
  static constexpr int B_STAGE_BYTES = BN * BK * 2;                // 16 KB
  static constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
  static constexpr int STG_BYTES = HEAD ? 0 : kWarps * 2 * 2048;   // bulk-store staging
  static constexpr int XBUF_BYTES = 2 * P * 128 * 8;               // (mean, M2), two parities
  static constexpr int HBUF_BYTES = HEAD ? 2 * P * 128 * NAP * 4 : 0;
  static constexpr int WEFF_BYTES = HEAD ? BN * NAP * 4 : 0;
  static constexpr int PAR_BYTES = 3 * BN * 4;                      // bias, gamma, beta of the slice
  static constexpr int EXTRA = STG_BYTES + XBUF_BYTES + HBUF_BYTES + WEFF_BYTES + PAR_BYTES + 1024 + 512;
  static constexpr int STAGES_FIT = (227 * 1024 - EXTRA) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_FIT > 6 ? 6 : STAGES_FIT;
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + EXTRA;
  static constexpr int TMEM_COLS = 2 * BN;
  static_assert(STAGES >= 2 && SMEM_BYTES <= 232448, "shared memory");
};

template <int CS, bool HEAD, bool PING>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_ln_cluster_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                           const __grid_constant__ CUtensorMap tmO, const EpiArgs e) {
  using S = LnShape<CS, HEAD, PING>;
  constexpr int NAP = S::NAP, P = S::P;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = sA + S::STAGES * A_STAGE_BYTES;
  uint8_t* s_stage = sB + S::STAGES * S::B_STAGE_BYTES;
  float2* xbuf = reinterpret_cast<float2*>(s_stage + S::STG_BYTES);                 // [2][P][128]
  float* hbuf = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(xbuf) + S::XBUF_BYTES);  // [2][P][128][NAP]
  float* s_weff = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(hbuf) + S::HBUF_BYTES);
  float* s_par = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(s_weff) + S::WEFF_BYTES);   // [3][BN]
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(s_par) + S::PAR_BYTES);
  uint64_t* empty = full + S::STAGES;
  uint64_t* acc_full = empty + S::STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* xfull = acc_empty + 2;    // [2][4]: statistics of lane quarter q have arrived
  uint64_t* hfull = xfull + 8;        // [2][4]: head partials have arrived (rank 0)
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(hfull + 8);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rk = cluster_rank();
  const int cid = blockIdx.x / CS, ncl = gridDim.x / CS;
  const int m_tiles = (e.M + BM - 1) / BM;
  const int my_tiles = m_tiles > cid ? (m_tiles - 1 - cid) / ncl + 1 : 0;   // equal within a cluster
  const int n0 = static_cast<int>(rk) * BN;
  const int num_kb = e.K / BK;
  constexpr uint16_t kAllCtas = static_cast<uint16_t>((1u << CS) - 1);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S::STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, CS);          // released by the MMAs of every CTA of the cluster
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full + b, 1);
      mbar_init(acc_empty + b, PING ? kGroupWarps : kWarps);
    }
    for (int i = 0; i < 8; ++i) {
      // PING: the waiting warp's expect_tx is the one arrival; the peers'
      // statistics complete as transaction bytes
      mbar_init(xfull + i, PING ? 1 : P * 32);
      mbar_init(hfull + i, P * 32);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc(tmem_holder, S::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  cluster_sync();                     // every CTA's barriers exist before any peer arrives
  pdl_launch_dependents();
  // the weights are not written by the preceding kernels: the weight part of
  // the first k-blocks is fetched before the wait (overlapping the
  // predecessor's tail); the activations only after it
  const int n_pre = my_tiles > 0 ? (num_kb < S::STAGES ? num_kb : S::STAGES) : 0;
  if (warp == 0 && lane == 0) {
    for (int kb = 0; kb < n_pre; ++kb) {   // fresh ring: these stages are free
      mbar_expect_tx(full + kb, S::STAGE_BYTES);
      tma_load_2d(sB + kb * S::B_STAGE_BYTES, &tmB, full + kb, kb * BK, n0);
    }
  }
  pdl_wait();
  if constexpr (HEAD) {
    for (int i = threadIdx.x; i < BN * NAP; i += NUM_THREADS) {
      const int c = i / NAP, a = i - c * NAP;
      s_weff[i] = a < e.n_act ? e.weff_z[static_cast<long long>(n0 + c) * e.n_act + a] : 0.f;
    }
  }
  for (int i = threadIdx.x; i < BN; i += NUM_THREADS) {
    s_par[i] = e.bias[n0 + i];
    s_par[BN + i] = e.gamma[n0 + i];
    s_par[2 * BN + i] = e.beta[n0 + i];
  }
  __syncthreads();

  if (warp == 0) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const int m0 = (cid + i * ncl) * BM;
        // every CTA of the cluster reads the same activation rows: each loads
        // BM / CS of them into the stage of all CTAs (multicast)
        const int a_rows = m0 + static_cast<int>(rk) * (BM / CS);
        uint8_t* a_dst = sA + static_cast<int>(rk) * (A_STAGE_BYTES / CS);
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % S::STAGES;
          if (it < n_pre) {     // weights in flight since before the wait
            tma_load_2d_mc(a_dst + s * A_STAGE_BYTES, &tmA, full + s, kb * BK, a_rows, kAllCtas);
            continue;
          }
          // the stage is free in every CTA of the cluster
          if (!mbar_wait(empty + s, ((it / S::STAGES) & 1) ^ 1, abort_flag)) {
            ok = false;
            break;
          }
          mbar_expect_tx(full + s, S::STAGE_BYTES);
          tma_load_2d_mc(a_dst + s * A_STAGE_BYTES, &tmA, full + s, kb * BK, a_rows, kAllCtas);
          tma_load_2d(sB + s * S::B_STAGE_BYTES, &tmB, full + s, kb * BK, n0);
        }
      }
      if (*abort_flag)
        for (int k = it > S::STAGES ? it - S::STAGES : 0; k < it; ++k)
          mbar_wait_plain(full + k % S::STAGES, (k / S::STAGES) & 1);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN);
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const int buf = i & 1;
        if (!mbar_wait(acc_empty + buf, ((i >> 1) & 1) ^ 1, abort_flag)) break;
        tc_fence_after();
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % S::STAGES;
          if (!mbar_wait(full + s, (it / S::STAGES) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t adesc = sdesc_sw128(smem_u32(sA + s * A_STAGE_BYTES));
          const uint64_t bdesc = sdesc_sw128(smem_u32(sB + s * S::B_STAGE_BYTES));
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            mma_bf16(tmem + buf * BN, adesc + 2 * k, bdesc + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          mma_commit_mc(empty + s, kAllCtas);   // this CTA's reads of the stage are done, in every CTA
        }
        mma_commit(acc_full + buf);
      }
    }
  } else if constexpr (PING) {
    const int ew = warp - 2;
    const int grp = ew / kGroupWarps;  // tiles i with i % 2 == grp, TMEM buffer grp
    const int q = warp & 3;            // TMEM lane quarter
    const int trow = q * 32 + lane;
    uint8_t* stage = s_stage + ew * 4096;
    const float* s_bias = s_par;
    const float* s_gamma = s_par + BN;
    const float* s_beta = s_par + 2 * BN;
    int kchunk = 0;
    float v[32];
    for (int i = grp; i < my_tiles; i += 2) {
      const int buf = grp, pb = grp;
      const uint32_t use = static_cast<uint32_t>(i >> 1) & 1;
      const int m0 = (cid + i * ncl) * BM;
      const int row = m0 + trow;
      const bool valid = row < e.M;
      // the residual does not depend on the product: its first 64 columns are
      // fetched before waiting for the accumulator, the rest one chunk ahead
      const uint4* rp = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(e.res) +
                                                       (valid ? row : 0) * e.ldr + n0);
      uint4 rres[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) rres[k] = valid ? __ldg(rp + k) : make_uint4(0, 0, 0, 0);
      bool go = mbar_wait(acc_full + buf, use, abort_flag);
      go = __shfl_sync(0xffffffffu, go ? 1 : 0, 0) != 0;
      if (!go) break;
      tc_fence_after();
      const uint32_t tacc = tmem + buf * BN + (static_cast<uint32_t>(q * 32) << 16);
      // pass 1: v = acc + bias + residual, written back to TMEM; per chunk of
      // 32 columns its mean and squared deviations, merged over the chunks
      // (pairwise update; equal chunk sizes)
      float mean_p = 0.f, m2 = 0.f;
#pragma unroll
      for (int c = 0; c < BN; c += 32) {
        tmem_ld32(tacc + c, v);
        const int rb = (c / 8) & 7;            // residual registers of this chunk
        float sum = 0.f;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&rres[rb + k]);
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const float2 f = __bfloat1622float2(h2[t]);
            const int j = 8 * k + 2 * t;
            v[j] += s_bias[c + j] + f.x;
            v[j + 1] += s_bias[c + j + 1] + f.y;
            sum += v[j] + v[j + 1];
          }
        }
        if (c + 64 < BN) {                     // this chunk's registers now hold chunk c + 64
#pragma unroll
          for (int k = 0; k < 4; ++k) rres[rb + k] = valid ? __ldg(rp + (c + 64) / 8 + k) : make_uint4(0, 0, 0, 0);
        }
        const float mc = sum * (1.f / 32.f);
        float m2c = 0.f;
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const float t = v[k] - mc;
          m2c = fmaf(t, t, m2c);
        }
        tmem_st32(tacc + c, v);
        if (c == 0) {
          mean_p = mc;
          m2 = m2c;
        } else {
          // merge n_a = c columns (mean_p, m2) with 32 (mc, m2c)
          const float na = static_cast<float>(c), nt = na + 32.f;
          const float dlt = mc - mean_p;
          mean_p = fmaf(dlt, 32.f / nt, mean_p);
          m2 = m2 + m2c + dlt * dlt * (na * 32.f / nt);
        }
      }
      // publish (mean, M2) of these 128 columns to every CTA of the cluster:
      // this CTA's slot by a plain store (read back by this thread), the
      // peers' by asynchronous stores counted on their barriers
      {
        float2* mine = xbuf + (pb * P + static_cast<int>(rk)) * 128 + trow;
        *mine = make_float2(mean_p, m2);
#pragma unroll
        for (int pr = 0; pr < CS; ++pr)
          if (pr != static_cast<int>(rk))
            st_async_f32x2(map_peer(mine, pr), mean_p, m2, map_peer(xfull + pb * 4 + q, pr));
      }
      if (lane == 0) mbar_expect_tx(xfull + pb * 4 + q, (CS - 1) * 32 * 8);
      bool ok = mbar_wait_cluster(xfull + pb * 4 + q, use, abort_flag);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok) break;
      float mp[P];
      float mean = 0.f;
#pragma unroll
      for (int p = 0; p < P; ++p) {
        const float2 x = xbuf[(pb * P + p) * 128 + trow];
        mp[p] = x.x;
        mean += x.x;
        m2 = p == 0 ? x.y : m2 + x.y;
      }
      mean *= 1.f / P;
#pragma unroll
      for (int p = 0; p < P; ++p) {
        const float t = mp[p] - mean;
        m2 = fmaf(static_cast<float>(BN) * t, t, m2);
      }
      const float rstd = rsqrtf(m2 / static_cast<float>(BN * CS) + e.ln_eps);
      // pass 2: normalise; store, or the head's partial logits
      float lg[NAP];
#pragma unroll
      for (int a = 0; a < NAP; ++a) lg[a] = 0.f;
#pragma unroll
      for (int c = 0; c < BN; c += 32) {
        tmem_ld32(tacc + c, v);
#pragma unroll
        for (int k = 0; k < 32; ++k) v[k] = (v[k] - mean) * rstd * s_gamma[c + k] + s_beta[c + k];
        if constexpr (!HEAD) {
          __nv_bfloat16* out = valid ? static_cast<__nv_bfloat16*>(e.out) + row * e.ldo + n0 + c : nullptr;
          store_chunk(v, out, valid, true, &tmO, n0 + c, m0 + q * 32, stage, kchunk++, lane);
        } else {
          const float4* w4 = reinterpret_cast<const float4*>(s_weff + c * NAP);
#pragma unroll
          for (int k = 0; k < 32; ++k) {
            const float4 w = w4[k];
            lg[0] = fmaf(v[k], w.x, lg[0]);
            lg[1] = fmaf(v[k], w.y, lg[1]);
            lg[2] = fmaf(v[k], w.z, lg[2]);
            lg[3] = fmaf(v[k], w.w, lg[3]);
          }
        }
      }
      // every read of this accumulator is done
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty + buf);
      if constexpr (HEAD) {
        // partial logits of these 128 columns -> rank 0
        float* mine = hbuf + ((pb * P + static_cast<int>(rk)) * 128 + trow) * NAP;
        st_peer_f32x4(map_peer(mine, 0), lg[0], lg[1], lg[2], lg[3]);
        mbar_arrive_peer(map_peer(hfull + pb * 4 + q, 0));
        if (rk == 0) {
          ok = mbar_wait_cluster(hfull + pb * 4 + q, use, abort_flag);
          ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
          if (!ok) break;
          if (valid && row < e.n_cand_rows) {
            const int na = e.n_act;
            float t[NAP];
#pragma unroll
            for (int a = 0; a < NAP; ++a) t[a] = 0.f;
#pragma unroll
            for (int p = 0; p < P; ++p) {
              const float4 x = *reinterpret_cast<const float4*>(hbuf + ((pb * P + p) * 128 + trow) * NAP);
              t[0] += x.x; t[1] += x.y; t[2] += x.z; t[3] += x.w;
            }
            float mx = -INFINITY;
#pragma unroll
            for (int a = 0; a < NAP; ++a)
              if (a < na) {
                t[a] += __ldg(e.xlog + static_cast<long long>(row) * na + a);
                mx = fmaxf(mx, t[a]);
              }
            float ssum = 0.f, pe[NAP];
#pragma unroll
            for (int a = 0; a < NAP; ++a) {
              pe[a] = a < na ? expf(t[a] - mx) : 0.f;
              ssum += pe[a];
            }
            const float inv = 1.f / ssum;
#pragma unroll
            for (int a = 0; a < NAP; ++a)
              if (a < na) {
                e.logits[static_cast<long long>(row) * na + a] = t[a];
                if (e.probs) e.probs[static_cast<long long>(row) * na + a] = pe[a] * inv;
              }
          }
        }
      }
    }
    if (lane == 0) bulk_wait_all();
  } else {
    // few tiles per cluster: all eight warps on each tile, two per lane
    // quarter, each 64 of the CTA's 128 columns
    const int ew = warp - 2;
    const int q = warp & 3;            // TMEM lane quarter
    const int h = ew / 4;              // 64-column half of this CTA's slice
    const int c0 = h * 64;
    const int slot = static_cast<int>(rk) * 2 + h;
    const int trow = q * 32 + lane;
    uint8_t* stage = s_stage + ew * 4096;
    int kchunk = 0;
    float v[32];
    for (int i = 0; i < my_tiles; ++i) {
      const int buf = i & 1, pb = i & 1;
      const uint32_t use = static_cast<uint32_t>(i >> 1) & 1;
      const int m0 = (cid + i * ncl) * BM;
      const int row = m0 + trow;
      const bool valid = row < e.M;
      // the residual row does not depend on the product: fetch it before
      // waiting for the accumulator, so its DRAM latency overlaps the MMAs
      uint4 rres[8];
      {
        const uint4* rp = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(e.res) +
                                                         (valid ? row : 0) * e.ldr + n0 + c0);
#pragma unroll
        for (int k = 0; k < 8; ++k) rres[k] = valid ? __ldg(rp + k) : make_uint4(0, 0, 0, 0);
      }
      bool go = mbar_wait(acc_full + buf, use, abort_flag);
      go = __shfl_sync(0xffffffffu, go ? 1 : 0, 0) != 0;
      if (!go) break;
      tc_fence_after();
      const uint32_t tacc = tmem + buf * BN + (static_cast<uint32_t>(q * 32) << 16) + c0;
      // pass 1: v = acc + bias + residual, written back to TMEM
      float sum = 0.f;
#pragma unroll
      for (int c = 0; c < 64; c += 32) {
        tmem_ld32(tacc + c, v);
        float b[32], r[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) b[k] = s_par[c0 + c + k];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&rres[c / 8 + k]);
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const float2 f = __bfloat1622float2(h2[t]);
            r[8 * k + 2 * t] = f.x;
            r[8 * k + 2 * t + 1] = f.y;
          }
        }
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          v[k] += b[k] + r[k];
          sum += v[k];
        }
        tmem_st32(tacc + c, v);
      }
      const float mean_p = sum * (1.f / 64.f);
      float m2 = 0.f;
#pragma unroll
      for (int c = 0; c < 64; c += 32) {
        tmem_ld32(tacc + c, v);
#pragma unroll
        for (int k = 0; k < 32; ++k) {
          const float t = v[k] - mean_p;
          m2 = fmaf(t, t, m2);
        }
      }
      // publish (mean, M2) of these 64 columns to every CTA of the cluster
      {
        float2* mine = xbuf + (pb * P + slot) * 128 + trow;
#pragma unroll
        for (int pr = 0; pr < CS; ++pr) {
          st_peer_f32x2(map_peer(mine, pr), mean_p, m2);
          mbar_arrive_peer(map_peer(xfull + pb * 4 + q, pr));
        }
      }
      bool ok = mbar_wait_cluster(xfull + pb * 4 + q, use, abort_flag);
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      if (!ok) break;
      float mp[P];
      float mean = 0.f;
#pragma unroll
      for (int p = 0; p < P; ++p) {
        const float2 x = xbuf[(pb * P + p) * 128 + trow];
        mp[p] = x.x;
        mean += x.x;
        m2 = p == 0 ? x.y : m2 + x.y;
      }
      mean *= 1.f / P;
#pragma unroll
      for (int p = 0; p < P; ++p) {
        const float t = mp[p] - mean;
        m2 = fmaf(64.f * t, t, m2);
      }
      const float rstd = rsqrtf(m2 / static_cast<float>(BN * CS) + e.ln_eps);
      // pass 3: normalise; store, or the head's partial logits
      float lg[NAP];
#pragma unroll
      for (int a = 0; a < NAP; ++a) lg[a] = 0.f;
#pragma unroll
      for (int c = 0; c < 64; c += 32) {
        tmem_ld32(tacc + c, v);
#pragma unroll
        for (int k = 0; k < 32; ++k) v[k] = (v[k] - mean) * rstd * s_par[BN + c0 + c + k] + s_par[2 * BN + c0 + c + k];
        if constexpr (!HEAD) {
          __nv_bfloat16* out = valid ? static_cast<__nv_bfloat16*>(e.out) + row * e.ldo + n0 + c0 + c : nullptr;
          store_chunk(v, out, valid, true, &tmO, n0 + c0 + c, m0 + q * 32, stage, kchunk++, lane);
        } else {
          const float4* w4 = reinterpret_cast<const float4*>(s_weff + (c0 + c) * NAP);
#pragma unroll
          for (int k = 0; k < 32; ++k) {
            const float4 w = w4[k];
            lg[0] = fmaf(v[k], w.x, lg[0]);
            lg[1] = fmaf(v[k], w.y, lg[1]);
            lg[2] = fmaf(v[k], w.z, lg[2]);
            lg[3] = fmaf(v[k], w.w, lg[3]);
          }
        }
      }
      if constexpr (HEAD) {
        // partial logits of these 64 columns -> rank 0
        float* mine = hbuf + ((pb * P + slot) * 128 + trow) * NAP;
        st_peer_f32x4(map_peer(mine, 0), lg[0], lg[1], lg[2], lg[3]);
        mbar_arrive_peer(map_peer(hfull + pb * 4 + q, 0));
        if (rk == 0 && h == 0) {
          ok = mbar_wait_cluster(hfull + pb * 4 + q, use, abort_flag);
          ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
          if (!ok) break;
          if (valid && row < e.n_cand_rows) {
            const int na = e.n_act;
            float t[NAP];
#pragma unroll
            for (int a = 0; a < NAP; ++a) t[a] = 0.f;
#pragma unroll
            for (int p = 0; p < P; ++p) {
              const float4 x = *reinterpret_cast<const float4*>(hbuf + ((pb * P + p) * 128 + trow) * NAP);
              t[0] += x.x; t[1] += x.y; t[2] += x.z; t[3] += x.w;
            }
            float mx = -INFINITY;
#pragma unroll
            for (int a = 0; a < NAP; ++a)
              if (a < na) {
                t[a] += __ldg(e.xlog + static_cast<long long>(row) * na + a);
                mx = fmaxf(mx, t[a]);
              }
            float ssum = 0.f, pe[NAP];
#pragma unroll
            for (int a = 0; a < NAP; ++a) {
              pe[a] = a < na ? expf(t[a] - mx) : 0.f;
              ssum += pe[a];
            }
            const float inv = 1.f / ssum;
#pragma unroll
            for (int a = 0; a < NAP; ++a)
              if (a < na) {
                e.logits[static_cast<long long>(row) * na + a] = t[a];
                if (e.probs) e.probs[static_cast<long long>(row) * na + a] = pe[a] * inv;
              }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty + buf);
    }
    if (lane == 0) bulk_wait_all();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();                     // no CTA leaves while a peer may still write into it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, S::TMEM_COLS);
  }
  if (threadIdx.x == 0 && *abort_flag) latch_status(e.status, TXS_ERR_DEVICE_TIMEOUT);
}

// ------------------------------------------------------------------ CTA pairs

// Rows of d = 256 NP columns on clusters of NP CTA pairs (HEAD: the last
// layer, whose LN output goes into the action head instead of memory):
// pair p computes columns [256 p, 256 p + 256) of a 256-row tile with
// M = 256 MMAs (cta_group::2), issued by its even CTA; CTA 2 p + r holds rows
// [128 r, 128 r + 128) of the tile in its TMEM (two 256-column buffers).
// Each CTA stages its 128 activation rows and 128 of its pair's 256 weight
// rows (32 KB per stage).  The row statistics of a CTA's 256 columns go to
// the CTA of the other pair that holds the same rows (st.async, counted on
// its barrier); with NP = 1 the row is whole in one CTA.  The eight epilogue
// warps form two groups taking alternate tiles, as in the cluster kernel.
// With HEAD each CTA forms the partial logits z . W_eff_z of its 256 columns
// (at most 4 actions) and sends them to the CTA of pair 0 with the same rows,
// which adds the x part and writes logits and probabilities.
// With RS the residual rows come through shared memory: the epilogue warp of
// lane quarter q owns four 32-row x 64-column boxes (128-byte swizzle), and
// after adding box c of its tile it loads box c of the CTA's next tile (TMA),
// which the other group's warp of the same quarter reads; so every tile's
// residual is in flight while the previous tile's epilogue runs, at the
// price of two operand stages.
constexpr int PBN = 256;               // columns per CTA (and per pair)
constexpr int kResBox = 32 * 64 * 2;   // one residual box: 32 rows x 64 bf16 columns
constexpr int kResStagedMaxK = 1024;   // longest K that takes the shared-memory residual

template <int NP, bool HEAD, bool RS>
struct PairShape {
  static constexpr int CS = 2 * NP;
  static constexpr int NAP = 4;                                     // head actions padded to 4
  static constexpr int B_STAGE_BYTES = 128 * BK * 2;                // 16 KB
  static constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
  static constexpr int STG_BYTES = HEAD ? 0 : kWarps * 2048;        // one bulk-store buffer per warp
  static constexpr int XBUF_BYTES = 2 * NP * 128 * 8;               // (mean, M2) per column block, two parities
  static constexpr int HBUF_BYTES = HEAD ? 2 * NP * 128 * NAP * 4 : 0;   // partial logits per column block
  static constexpr int WEFF_BYTES = HEAD ? PBN * NAP * 4 : 0;
  static constexpr int PAR_BYTES = 3 * PBN * 4;
  static constexpr int RES_BYTES = RS ? 4 * (PBN / 64) * kResBox : 0;   // [quarter][box]
  static constexpr int EXTRA =
      RES_BYTES + STG_BYTES + XBUF_BYTES + HBUF_BYTES + WEFF_BYTES + PAR_BYTES + 1024 + 640;
  static constexpr int STAGES_FIT = (227 * 1024 - EXTRA) / STAGE_BYTES;
  static constexpr int STAGES = STAGES_FIT > 8 ? 8 : STAGES_FIT;
  static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + EXTRA;
  static constexpr int TMEM_COLS = 2 * PBN;
  static_assert(STAGES >= 4 && SMEM_BYTES <= 232448, "shared memory");
};

template <int NP, bool HEAD, bool RS>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_ln_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                        const __grid_constant__ CUtensorMap tmO, const __grid_constant__ CUtensorMap tmR,
                        const EpiArgs e) {
  using S = PairShape<NP, HEAD, RS>;
  constexpr int NAP = S::NAP;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = sA + S::STAGES * A_STAGE_BYTES;
  uint8_t* s_res = sB + S::STAGES * S::B_STAGE_BYTES;                                 // [4][PBN / 64] boxes
  uint8_t* s_stage = s_res + S::RES_BYTES;
  float2* xbuf = reinterpret_cast<float2*>(s_stage + S::STG_BYTES);                 // [2][NP][128]
  float* hbuf = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(xbuf) + S::XBUF_BYTES);     // [2][NP][128][NAP]
  float* s_weff = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(hbuf) + S::HBUF_BYTES);  // [PBN][NAP]
  float* s_par = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(s_weff) + S::WEFF_BYTES);  // [3][PBN]
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(s_par) + S::PAR_BYTES);
  uint64_t* empty = full + S::STAGES;
  uint64_t* acc_full = empty + S::STAGES;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* xfull = acc_empty + 2;    // [2][4]: the other pair's statistics of lane quarter q
  uint64_t* hfull = xfull + 8;        // [2][4]: the other pairs' partial logits (pair 0, HEAD)
  uint64_t* res_full = hfull + 8;     // [4][PBN / 64]: residual box landed (RS)
  int* res_iss = reinterpret_cast<int*>(res_full + 16);    // per box: last tile whose load was issued
  int* res_seen = res_iss + 16;                            // per box: last tile whose load was waited for
  uint32_t* tmem_holder = reinterpret_cast<uint32_t*>(res_seen + 16);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_holder + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rk = cluster_rank();
  const int pr = static_cast<int>(rk) >> 1, half = static_cast<int>(rk) & 1;
  const uint32_t lead_rank = rk & ~1u;
  const uint16_t pair_mask = static_cast<uint16_t>(3u << (2 * pr));
  const int cid = blockIdx.x / S::CS, ncl = gridDim.x / S::CS;
  const int m_tiles = (e.M + 2 * BM - 1) / (2 * BM);
  const int my_tiles = m_tiles > cid ? (m_tiles - 1 - cid) / ncl + 1 : 0;   // equal within a cluster
  const int n0 = pr * PBN;                      // this pair's columns
  const int nb0 = n0 + half * 128;              // this CTA's weight rows
  const int num_kb = e.K / BK;
  constexpr uint32_t kFullBytes = 2 * S::STAGE_BYTES;   // both CTAs' loads, on the even CTA's barrier

  if (threadIdx.x == 0) {
    for (int s = 0; s < S::STAGES; ++s) {
      mbar_init(full + s, 1);
      mbar_init(empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full + b, 1);
      mbar_init(acc_empty + b, 2 * kGroupWarps);     // the even CTA's: both CTAs' group
    }
    for (int i = 0; i < 8; ++i) {
      mbar_init(xfull + i, 1);
      mbar_init(hfull + i, 1);
    }
    for (int i = 0; i < 16; ++i) {
      mbar_init(res_full + i, 1);
      res_iss[i] = res_seen[i] = -1;
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) tmem_alloc_pair(tmem_holder, S::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_holder;
  cluster_sync();                     // every CTA's barriers exist before any peer signals them
  pdl_launch_dependents();
  auto lead = [&](uint64_t* bar) { return map_peer(bar, lead_rank); };
  const int n_pre = my_tiles > 0 ? (num_kb < S::STAGES ? num_kb : S::STAGES) : 0;
  if (warp == 0 && lane == 0) {
    for (int kb = 0; kb < n_pre; ++kb) {   // weights: not written by the preceding kernels
      if (half == 0) mbar_expect_tx(full + kb, kFullBytes);
      tma_load_2d_pair(sB + kb * S::B_STAGE_BYTES, &tmB, lead(full + kb), kb * BK, nb0);
    }
  }
  pdl_wait();
  for (int i = threadIdx.x; i < PBN; i += NUM_THREADS) {
    s_par[i] = e.bias[n0 + i];
    s_par[PBN + i] = e.gamma[n0 + i];
    s_par[2 * PBN + i] = e.beta[n0 + i];
  }
  if constexpr (HEAD) {
    for (int i = threadIdx.x; i < PBN * NAP; i += NUM_THREADS) {
      const int c = i / NAP, a = i - c * NAP;
      s_weff[i] = a < e.n_act ? e.weff_z[static_cast<long long>(n0 + c) * e.n_act + a] : 0.f;
    }
  }
  __syncthreads();

  if (warp == 0) {
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const int a_rows = (cid + i * ncl) * 2 * BM + half * BM;
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % S::STAGES;
          if (it < n_pre) {     // weights in flight since before the wait
            tma_load_2d_pair(sA + s * A_STAGE_BYTES, &tmA, lead(full + s), kb * BK, a_rows);
            continue;
          }
          if (!mbar_wait(empty + s, ((it / S::STAGES) & 1) ^ 1, abort_flag)) {
            ok = false;
            break;
          }
          if (half == 0) mbar_expect_tx(full + s, kFullBytes);
          tma_load_2d_pair(sA + s * A_STAGE_BYTES, &tmA, lead(full + s), kb * BK, a_rows);
          tma_load_2d_pair(sB + s * S::B_STAGE_BYTES, &tmB, lead(full + s), kb * BK, nb0);
        }
      }
      // the pair's MMAs release this CTA's stages by multicast commits: take
      // the last ones before the CTA may exit
      for (int k = it > S::STAGES ? it - S::STAGES : 0; k < it && !*abort_flag; ++k)
        mbar_wait(empty + k % S::STAGES, (k / S::STAGES) & 1, abort_flag);
      if (*abort_flag && half == 0)
        for (int k = it > S::STAGES ? it - S::STAGES : 0; k < it; ++k)
          mbar_wait_plain(full + k % S::STAGES, (k / S::STAGES) & 1);
    }
  } else if (warp == 1) {
    if (lane == 0 && half == 0) {
      constexpr uint32_t idesc = idesc_bf16(2 * BM, PBN);
      int it = 0;
      bool ok = true;
      for (int i = 0; i < my_tiles && ok; ++i) {
        const int buf = i & 1;
        if (!mbar_wait(acc_empty + buf, ((i >> 1) & 1) ^ 1, abort_flag)) break;
        tc_fence_after();
        for (int kb = 0; kb < num_kb; ++kb, ++it) {
          const int s = it % S::STAGES;
          if (!mbar_wait(full + s, (it / S::STAGES) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t adesc = sdesc_sw128(smem_u32(sA + s * A_STAGE_BYTES));
          const uint64_t bdesc = sdesc_sw128(smem_u32(sB + s * S::B_STAGE_BYTES));
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            mma_bf16_pair(tmem + buf * PBN, adesc + 2 * k, bdesc + 2 * k, idesc, (kb > 0 || k > 0) ? 1u : 0u);
          mma_commit_pair(empty + s, pair_mask);
        }
        mma_commit_pair(acc_full + buf, pair_mask);   // also on abort: the epilogues wait on every issued MMA
      }
    }
  } else {
    const int ew = warp - 2;
    const int grp = ew / kGroupWarps;  // tiles i with i % 2 == grp, TMEM buffer grp
    const int q = warp & 3;            // TMEM lane quarter
    const int trow = q * 32 + lane;
    uint8_t* stage = s_stage + ew * 2048;
    const float* s_bias = s_par;
    const float* s_gamma = s_par + PBN;
    const float* s_beta = s_par + 2 * PBN;
    int kchunk = 0;
    float v[32];
    // RS: this quarter's residual boxes; lane 0 loads box c of the rows of
    // this CTA's tile j (rows past M read as zeros)
    constexpr int kBoxes = PBN / 64;
    uint8_t* res_q = s_res + q * kBoxes * kResBox;
    uint64_t* res_bar = res_full + q * kBoxes;
    auto res_issue = [&](int j, int c) {
      mbar_expect_tx(res_bar + c, kResBox);
      tma_load_2d(res_q + c * kResBox, &tmR, res_bar + c, n0 + 64 * c, (cid + j * ncl) * 2 * BM + half * BM + q * 32);
      res_iss[q * kBoxes + c] = j;
    };
    if constexpr (RS) {
      // the first tile's boxes; later ones are loaded by the previous tile's warp
      if (grp == 0 && lane == 0 && my_tiles > 0)
        for (int c = 0; c < kBoxes; ++c) res_issue(0, c);
    }
    for (int i = grp; i < my_tiles; i += 2) {
      const int buf = grp, pb = grp;
      const uint32_t use = static_cast<uint32_t>(i >> 1) & 1;
      const int m0 = (cid + i * ncl) * 2 * BM + half * BM;   // this CTA's rows
      const int row = m0 + trow;
      const bool valid = row < e.M;
      // without RS the residual's first 64 columns are fetched before the
      // wait, the rest one chunk ahead
      const uint4* rp = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(e.res) +
                                                       static_cast<long long>(valid ? row : 0) * e.ldr + n0);
      uint4 rres[8];
      if constexpr (!RS) {
#pragma unroll
        for (int k = 0; k < 8; ++k) rres[k] = valid ? __ldg(rp + k) : make_uint4(0, 0, 0, 0);
      }
      bool go = mbar_wait(acc_full + buf, use, abort_flag);
      go = __shfl_sync(0xffffffffu, go ? 1 : 0, 0) != 0;
      if (!go) break;
      tc_fence_after();
      const uint32_t tacc = tmem + buf * PBN + (static_cast<uint32_t>(q * 32) << 16);
      // pass 1: v = acc + bias + residual, written back to TMEM; per chunk of
      // 32 columns its mean and squared deviations, merged pairwise
      float mean_p = 0.f, m2 = 0.f;
      // 64 columns per iteration: chunk h of 32 uses residual registers
      // rres[4 h .. 4 h + 3] (static indices), then refills them for c + 64
      // (RS: box c64 / 64 read from shared memory when it has landed)
      bool res_ok = true;
#pragma unroll 1
      for (int c64 = 0; c64 < PBN; c64 += 64) {
        if constexpr (RS) {
          const int cb = c64 / 64;
          res_ok = mbar_wait(res_bar + cb, static_cast<uint32_t>(i) & 1, abort_flag);
          res_ok = __shfl_sync(0xffffffffu, res_ok ? 1 : 0, 0) != 0;
          if (!res_ok) break;
          if (lane == 0) res_seen[q * kBoxes + cb] = i;
          const uint8_t* bx = res_q + cb * kResBox + lane * 128;
#pragma unroll
          for (int k = 0; k < 8; ++k) rres[k] = *reinterpret_cast<const uint4*>(bx + ((k ^ (lane & 7)) << 4));
        }
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int c = c64 + 32 * hh;
          tmem_ld32(tacc + c, v);
          float sum = 0.f;
          const float4* b4 = reinterpret_cast<const float4*>(s_bias + c);   // broadcast 16-byte reads
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&rres[4 * hh + k]);
            const float4 bl = b4[2 * k], bh = b4[2 * k + 1];
            const float bk[8] = {bl.x, bl.y, bl.z, bl.w, bh.x, bh.y, bh.z, bh.w};
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const float2 f = __bfloat1622float2(h2[t]);
              const int j = 8 * k + 2 * t;
              v[j] += bk[2 * t] + f.x;
              v[j + 1] += bk[2 * t + 1] + f.y;
              sum += v[j] + v[j + 1];
            }
          }
          if (!RS && c + 64 < PBN) {
#pragma unroll
            for (int k = 0; k < 4; ++k)
              rres[4 * hh + k] = valid ? __ldg(rp + (c + 64) / 8 + k) : make_uint4(0, 0, 0, 0);
          }
          const float mc = sum * (1.f / 32.f);
          float m2c = 0.f;
#pragma unroll
          for (int k = 0; k < 32; ++k) {
            const float t = v[k] - mc;
            m2c = fmaf(t, t, m2c);
          }
          tmem_st32(tacc + c, v);
          if (c == 0) {
            mean_p = mc;
            m2 = m2c;
          } else {
            const float na = static_cast<float>(c), nt = na + 32.f;
            const float dlt = mc - mean_p;
            mean_p = fmaf(dlt, 32.f / nt, mean_p);
            m2 = m2 + m2c + dlt * dlt * (na * 32.f / nt);
          }
        }
        if constexpr (RS) {
          // every lane has consumed the box: the next tile's rows go into it
          fence_async_smem();
          __syncwarp();
          if (lane == 0 && i + 1 < my_tiles) res_issue(i + 1, c64 / 64);
        }
      }
      if (!res_ok) break;
      float mean = mean_p;
      if constexpr (NP > 1) {
        // (mean, M2) of these 256 columns to the CTAs of the other pairs that
        // hold the same rows; this CTA's own slot by a plain store
        float2* mine = xbuf + (pb * NP + pr) * 128 + trow;
        *mine = make_float2(mean_p, m2);
#pragma unroll
        for (int o = 0; o < NP; ++o)
          if (o != pr) {
            const uint32_t peer = static_cast<uint32_t>(2 * o + half);
            st_async_f32x2(map_peer(mine, peer), mean_p, m2, map_peer(xfull + pb * 4 + q, peer));
          }
        if (lane == 0) mbar_expect_tx(xfull + pb * 4 + q, (NP - 1) * 32 * 8);
        bool ok = mbar_wait_cluster(xfull + pb * 4 + q, use, abort_flag);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (!ok) break;
        float mp[NP];
        mean = 0.f;
#pragma unroll
        for (int o = 0; o < NP; ++o) {
          const float2 x = xbuf[(pb * NP + o) * 128 + trow];
          mp[o] = x.x;
          mean += x.x;
          m2 = o == 0 ? x.y : m2 + x.y;
        }
        mean *= 1.f / NP;
#pragma unroll
        for (int o = 0; o < NP; ++o) {
          const float t = mp[o] - mean;
          m2 = fmaf(static_cast<float>(PBN) * t, t, m2);
        }
      }
      const float rstd = rsqrtf(m2 / static_cast<float>(PBN * NP) + e.ln_eps);
      // pass 2: normalise and store, or the head's partial logits
      float lg[NAP];
#pragma unroll
      for (int a = 0; a < NAP; ++a) lg[a] = 0.f;
#pragma unroll 1
      for (int c = 0; c < PBN; c += 32) {
        tmem_ld32(tacc + c, v);
        const float4* g4 = reinterpret_cast<const float4*>(s_gamma + c);
        const float4* e4 = reinterpret_cast<const float4*>(s_beta + c);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const float4 g = g4[k], b = e4[k];
          v[4 * k] = (v[4 * k] - mean) * rstd * g.x + b.x;
          v[4 * k + 1] = (v[4 * k + 1] - mean) * rstd * g.y + b.y;
          v[4 * k + 2] = (v[4 * k + 2] - mean) * rstd * g.z + b.z;
          v[4 * k + 3] = (v[4 * k + 3] - mean) * rstd * g.w + b.w;
        }
        if constexpr (!HEAD) {
          __nv_bfloat16* out =
              valid ? static_cast<__nv_bfloat16*>(e.out) + static_cast<long long>(row) * e.ldo + n0 + c : nullptr;
          store_chunk<1>(v, out, valid, true, &tmO, n0 + c, m0 + q * 32, stage, kchunk++, lane);
        } else {
          const float4* w4 = reinterpret_cast<const float4*>(s_weff + c * NAP);
#pragma unroll
          for (int k = 0; k < 32; ++k) {
            const float4 w = w4[k];
            lg[0] = fmaf(v[k], w.x, lg[0]);
            lg[1] = fmaf(v[k], w.y, lg[1]);
            lg[2] = fmaf(v[k], w.z, lg[2]);
            lg[3] = fmaf(v[k], w.w, lg[3]);
          }
        }
      }
      // every read of this accumulator is done: release it on the even CTA
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_peer_signal(lead(acc_empty + buf));
      if constexpr (HEAD) {
        // partial logits of these 256 columns -> the CTA of pair 0 with the same rows
        float* mine = hbuf + ((pb * NP + pr) * 128 + trow) * NAP;
        if (pr == 0) {
          *reinterpret_cast<float4*>(mine) = make_float4(lg[0], lg[1], lg[2], lg[3]);
        } else {
          const uint32_t owner = static_cast<uint32_t>(half);
          st_async_f32x4(map_peer(mine, owner), lg[0], lg[1], lg[2], lg[3], map_peer(hfull + pb * 4 + q, owner));
        }
        if (pr == 0) {
          if constexpr (NP > 1) {
            if (lane == 0) mbar_expect_tx(hfull + pb * 4 + q, (NP - 1) * 32 * NAP * 4);
            bool ok = mbar_wait_cluster(hfull + pb * 4 + q, use, abort_flag);
            ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
            if (!ok) break;
          }
          if (valid && row < e.n_cand_rows) {
            const int na = e.n_act;
            float t[NAP];
#pragma unroll
            for (int a = 0; a < NAP; ++a) t[a] = 0.f;
#pragma unroll
            for (int o = 0; o < NP; ++o) {
              const float4 x = *reinterpret_cast<const float4*>(hbuf + ((pb * NP + o) * 128 + trow) * NAP);
              t[0] += x.x; t[1] += x.y; t[2] += x.z; t[3] += x.w;
            }
            float mx = -INFINITY;
#pragma unroll
            for (int a = 0; a < NAP; ++a)
              if (a < na) {
                t[a] += __ldg(e.xlog + static_cast<long long>(row) * na + a);
                mx = fmaxf(mx, t[a]);
              }
            float ssum = 0.f, pe[NAP];
#pragma unroll
            for (int a = 0; a < NAP; ++a) {
              pe[a] = a < na ? expf(t[a] - mx) : 0.f;
              ssum += pe[a];
            }
            const float inv = 1.f / ssum;
#pragma unroll
            for (int a = 0; a < NAP; ++a)
              if (a < na) {
                e.logits[static_cast<long long>(row) * na + a] = t[a];
                if (e.probs) e.probs[static_cast<long long>(row) * na + a] = pe[a] * inv;
              }
          }
        }
      }
    }
    if (lane == 0) bulk_wait_all();
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (RS) {
    // after an abort: a residual box whose load was issued but never waited
    // for lands before the CTA exits
    if (threadIdx.x < 16 && *abort_flag && res_iss[threadIdx.x] > res_seen[threadIdx.x])
      mbar_wait_plain(res_full + threadIdx.x, static_cast<uint32_t>(res_iss[threadIdx.x]) & 1);
    __syncthreads();
  }
  cluster_sync();                     // no CTA leaves while a peer may still signal or write into it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem, S::TMEM_COLS);
  }
  if (threadIdx.x == 0 && *abort_flag) latch_status(e.status, TXS_ERR_DEVICE_TIMEOUT);
}

template <int NP, bool HEAD, bool RS>
static cudaError_t launch_pair(const __nv_bfloat16* A, long long lda, const __nv_bfloat16* B, const EpiArgs& e,
                               cudaStream_t s, int cls) {
  using Sh = PairShape<NP, HEAD, RS>;
  auto kern = gemm_ln_pair_kernel<NP, HEAD, RS>;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = Sh::CS;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = Sh::SMEM_BYTES;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  static int max_clusters = 0;
  if (!max_clusters) {
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Sh::SMEM_BYTES);
    if (err != cudaSuccess) return err;
    cfg.gridDim = dim3((num_sms() / Sh::CS) * Sh::CS);
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n <= 0) {
      (void)cudaGetLastError();
      n = num_sms() / Sh::CS;
    }
    max_clusters = n;
  }
  CUtensorMap ta, tb, to, tr;
  if (!make_tmap(&ta, A, e.M, e.K, lda, BM)) return cudaErrorInvalidValue;
  if (!make_tmap(&tb, B, e.N, e.K, e.K, 128)) return cudaErrorInvalidValue;
  if (HEAD) to = ta;   // unused
  else if (!make_tmap_out(&to, e.out, e.M, e.N, e.ldo)) return cudaErrorInvalidValue;
  // residual boxes of 32 rows x 64 columns (RS)
  if (!RS) tr = ta;   // unused
  else if (!make_tmap(&tr, e.res, e.M, e.N, e.ldr, 32)) return cudaErrorInvalidValue;
  const int m_tiles = (e.M + 2 * BM - 1) / (2 * BM);
  const int ncl = m_tiles < max_clusters ? m_tiles : max_clusters;
  cfg.gridDim = dim3(ncl * Sh::CS);
  cfg.numAttrs = 2;
  prof_begin(cls, s);
  cudaError_t err = cudaLaunchKernelEx(&cfg, kern, ta, tb, to, tr, e);
  prof_end(cls, s);
  return err;
}

template <int CS, bool HEAD, bool PING>
static cudaError_t launch_cs(const __nv_bfloat16* A, long long lda, const __nv_bfloat16* B, const EpiArgs& e,
                             cudaStream_t s, int cls) {
  using Sh = LnShape<CS, HEAD, PING>;
  auto kern = gemm_ln_cluster_kernel<CS, HEAD, PING>;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = CS;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = Sh::SMEM_BYTES;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // clusters that can be resident at once (one CTA per SM)
  static int max_clusters = 0;
  if (!max_clusters) {
    cudaError_t err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, Sh::SMEM_BYTES);
    if (err != cudaSuccess) return err;
    cfg.gridDim = dim3((num_sms() / CS) * CS);
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n <= 0) {
      (void)cudaGetLastError();
      n = num_sms() / CS;
    }
    max_clusters = n;
  }
  CUtensorMap ta, tb, to;
  // activation boxes of BM / CS rows: each CTA multicasts its share of a tile
  if (!make_tmap(&ta, A, e.M, e.K, lda, BM / CS)) return cudaErrorInvalidValue;
  if (!make_tmap(&tb, B, e.N, e.K, e.K, BN)) return cudaErrorInvalidValue;
  if (HEAD) to = ta;   // unused
  else if (!make_tmap_out(&to, e.out, e.M, e.N, e.ldo)) return cudaErrorInvalidValue;
  const int m_tiles = (e.M + BM - 1) / BM;
  const int ncl = m_tiles < max_clusters ? m_tiles : max_clusters;
  cfg.gridDim = dim3(ncl * CS);
  cfg.numAttrs = 2;
  prof_begin(cls, s);
  cudaError_t err = cudaLaunchKernelEx(&cfg, kern, ta, tb, to, e);
  prof_end(cls, s);
  return err;
}

}  // namespace tcln

namespace tc {

cudaError_t launch_gemm_ln_cluster(const __nv_bfloat16* A, long long lda, const __nv_bfloat16* B, const EpiArgs& e,
                                   cudaStream_t s, int cls) {
  if (e.epi == EPI_LN_HEAD && (e.n_act < 1 || e.n_act > 4)) return cudaErrorNotSupported;
  if (e.epi != EPI_LN && e.epi != EPI_LN_HEAD) return cudaErrorNotSupported;
  const bool head = e.epi == EPI_LN_HEAD;
  // CTA pairs (256 columns per CTA) once every cluster gets two 256-row tiles
  if ((e.N == 256 || e.N == 512) && (!head || e.n_act <= 4)) {
    const int ncs = e.N / 128;   // CTAs per cluster either way
    if ((e.M + 2 * tc::BM - 1) / (2 * tc::BM) >= 2 * (num_sms() / ncs)) {
      if (head)
        return e.N == 256 ? tcln::launch_pair<1, true, false>(A, lda, B, e, s, cls)
                          : tcln::launch_pair<2, true, false>(A, lda, B, e, s, cls);
      // short K: the residual through shared memory (the mainloop keeps
      // up with four operand stages); long K keeps six stages
      if (e.K <= tcln::kResStagedMaxK)
        return e.N == 256 ? tcln::launch_pair<1, false, true>(A, lda, B, e, s, cls)
                          : tcln::launch_pair<2, false, true>(A, lda, B, e, s, cls);
      return e.N == 256 ? tcln::launch_pair<1, false, false>(A, lda, B, e, s, cls)
                        : tcln::launch_pair<2, false, false>(A, lda, B, e, s, cls);
    }
  }
  // the two epilogue groups pay off once each cluster has several row tiles
  const int m_tiles = (e.M + tc::BM - 1) / tc::BM;
  const bool ping = m_tiles >= 4 * (num_sms() / (e.N / tcln::BN));
  switch (e.N) {
    case 256:
      if (ping) return head ? tcln::launch_cs<2, true, true>(A, lda, B, e, s, cls)
                            : tcln::launch_cs<2, false, true>(A, lda, B, e, s, cls);
      return head ? tcln::launch_cs<2, true, false>(A, lda, B, e, s, cls)
                  : tcln::launch_cs<2, false, false>(A, lda, B, e, s, cls);
    case 512:
      if (ping) return head ? tcln::launch_cs<4, true, true>(A, lda, B, e, s, cls)
                            : tcln::launch_cs<4, false, true>(A, lda, B, e, s, cls);
      return head ? tcln::launch_cs<4, true, false>(A, lda, B, e, s, cls)
                  : tcln::launch_cs<4, false, false>(A, lda, B, e, s, cls);
    default: return cudaErrorNotSupported;
  }
}

}  // namespace tc
}  // namespace txs
