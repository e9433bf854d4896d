// The question's forward through the shallow layers (Sec. 4.2, Eq. 10).
//
// Eq. 10 appends the question to the retained shallow history and runs it through layers
// [0, P); layer i's attention reads the layer's stored keys and values, and the layer
// yields the question's query states Q^i, which the retrieval scores (Eq. 11). The
// backbone is synthetic: pre-norm GQA decoder layers (RMSNorm, q/k/v projections with
// bias, rotate-half RoPE, attention, output projection, SwiGLU MLP, residual adds).
// Rounding points: the operands of every matrix product and the outputs q, k, v are
// bf16 (nearest-even); the hidden states H stay fp32.
//
// Kernels per layer (R question rows, Rp = R rounded up to 16):
//   k_fw_norm     H (+)= the split-K partial sums of the previous product (fixed order),
//                 then X = bf16(RMSNorm(H) * w)
//   k_fw_gemm     partial[split] = X W^T on the tcgen05 tensor cores: 128 output features
//                 of W on the TMEM lanes (A operand), the Rp rows as N, K split over CTAs;
//                 W and X tiles by TMA (128-byte swizzle) through a ring of stages
//   k_fw_qkv      q, k, v from the partials (+ bias), RoPE on q and k with exact (fp64)
//                 angles; q goes to the caller's Q^i
//   k_fw_attn     the question rows of one key head against a chunk of the layer's
//                 stored tokens: S = Q K^T (rows on the TMEM lanes), P = 2^(s - m) in bf16,
//                 O += P V on the tensor cores, with the running max raised lazily (only
//                 when a tile's max exceeds it by 8, scaling O and l then); per chunk the
//                 unnormalised (m, l, O)
//   k_fw_attn_out the chunks and the question's own rows (causal) merged per (row, head)
//                 in a fixed order, o = bf16(O / L)
//   k_fw_swiglu   a = bf16(silu(g) * u) from the gate and up partials
#include "ss_internal.cuh"
#include "ss_device.cuh"
#include "ss_tc.cuh"
#include "ss_pack.cuh"

#include <algorithm>

namespace ss {

// Bounded wait that gives up when another role of the CTA raised the abort flag; a wait
// that runs out raises it.
__device__ __forceinline__ bool fw_wait(uint32_t bar, uint32_t parity, volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (uint32_t i = 1; i < kDefaultWaitPolls; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255u) == 0u) {
      if (*abort) return false;
      if (global_ns() - t0 > 1000000000ull) break;
    }
  }
  *abort = 1;
  return false;
}

__device__ __forceinline__ void fw_bar(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// ===========================================================================
// Skinny GEMM: part[split][r][n] = sum over the split's K range of X[r][k] W[n][k].
// With swiglu_I > 0 (one split), the gate/up projection with the MLP's product fused: CTA b
// stages gate rows 64 b .. 64 b + 63 of W (TMEM lanes 0-63) and the matching up rows
// I + 64 b .. (lanes 64-127) as one 128-row operand, and its epilogue writes
// A[r][f] = bf16(silu(g) * u) directly (no partials, no separate kernel).
// ===========================================================================
constexpr int kGmThreads = 192;           // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr int kGmMaxStages = 8;
constexpr int kGmABytes = 128 * 128;      // 128 rows of W x 64 bf16

struct GemmJob {
  float* part;       // [splits][Rp][n_out]
  int n_out;
  int swiglu_I;      // > 0: gate/up with SwiGLU in the epilogue (splits 1; see below)
  __nv_bfloat16* A;  // [Rp][swiglu_I] the SwiGLU product (rows >= R zero)
  int R, Rp;
  int kblocks;       // K / 64
  int splits;
  int stages;
  uint32_t* status;
};

struct GmBars {
  unsigned long long full[kGmMaxStages], empty[kGmMaxStages], d_full;
  uint32_t taddr;
  int abort;
};

__global__ void __launch_bounds__(kGmThreads, 1)
    k_fw_gemm(const __grid_constant__ CUtensorMap wmap, const __grid_constant__ CUtensorMap xmap,
              const GemmJob J) {
  extern __shared__ unsigned char sm_raw[];
  __shared__ GmBars S;
  unsigned char* sm = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(sm_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int stages = J.stages;
  const int b_bytes = J.Rp * 128;
  const int stage_bytes = kGmABytes + b_bytes;   // a multiple of 1024 (Rp % 16 == 0)
  const int m0 = blockIdx.x * (J.swiglu_I > 0 ? 64 : 128), split = blockIdx.y;
  const int kb0 = (int)((int64_t)J.kblocks * split / J.splits);
  const int kb1 = (int)((int64_t)J.kblocks * (split + 1) / J.splits);
  const int n = kb1 - kb0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort = &S.abort;
  if (threadIdx.x == 0) {
    for (int s = 0; s < stages; ++s) {
      mbar_init(smem_u32(&S.full[s]), 1);
      mbar_init(smem_u32(&S.empty[s]), 1);
    }
    mbar_init(smem_u32(&S.d_full), 1);
    S.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&S.taddr), 64);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_release();
  const uint32_t tbase = S.taddr;
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&wmap);
    tma_prefetch_map(&xmap);
    int issued_last[kGmMaxStages];
    for (int s = 0; s < kGmMaxStages; ++s) issued_last[s] = -1;
    // the weights do not depend on the previous kernel: the first stages' weight tiles
    // are requested before waiting for it, their rows of X after
    const int pre = n < stages ? n : stages;
    // W rows of a stage: 128 from m0, or 64 gate rows from m0 and 64 up rows from I + m0
    auto load_w = [&](uint32_t dst, uint32_t bar, int kx) {
      if (J.swiglu_I > 0) {
        tma_load_2d(dst, &wmap, bar, kx, m0);
        tma_load_2d(dst + kGmABytes / 2, &wmap, bar, kx, J.swiglu_I + m0);
      } else {
        tma_load_2d(dst, &wmap, bar, kx, m0);
      }
    };
    for (int j = 0; j < pre; ++j) {
      const uint32_t bar = smem_u32(&S.full[j]);
      mbar_expect_tx(bar, (uint32_t)stage_bytes);
      load_w(smem_u32(sm + j * stage_bytes), bar, (kb0 + j) * 64);
    }
    pdl_wait();
    for (int j = 0; j < pre; ++j) {
      tma_load_2d(smem_u32(sm + j * stage_bytes) + kGmABytes, &xmap, smem_u32(&S.full[j]),
                  (kb0 + j) * 64, 0);
      issued_last[j] = j;
    }
    for (int j = pre; j < n && !*abort; ++j) {
      const int st = j % stages;
      if (!fw_wait(smem_u32(&S.empty[st]), ((j / stages) - 1) & 1, abort)) break;
      const uint32_t bar = smem_u32(&S.full[st]);
      const uint32_t dst = smem_u32(sm + st * stage_bytes);
      mbar_expect_tx(bar, (uint32_t)stage_bytes);
      load_w(dst, bar, (kb0 + j) * 64);
      tma_load_2d(dst + kGmABytes, &xmap, bar, (kb0 + j) * 64, 0);
      issued_last[st] = j;
    }
    // the copies in flight land before the CTA ends
    for (int s = 0; s < stages; ++s)
      if (issued_last[s] >= 0) mbar_wait_bounded(smem_u32(&S.full[s]), (issued_last[s] / stages) & 1);
  } else if (warp == 1 && lane == 0) {
    const uint32_t id = idesc_bf16_f32(128, J.Rp, false, false);
    for (int j = 0; j < n; ++j) {
      const int st = j % stages;
      if (!fw_wait(smem_u32(&S.full[st]), (j / stages) & 1, abort)) break;
      tc_fence_after();
      const uint32_t a = smem_u32(sm + st * stage_bytes);
      const uint32_t b = a + kGmABytes;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        umma_bf16(tbase, sdesc_sw128(a + k * 32, 16, 1024), sdesc_sw128(b + k * 32, 16, 1024), id,
                  (j > 0 || k > 0) ? 1u : 0u);
      umma_commit(smem_u32(&S.empty[st]));
    }
    umma_commit(smem_u32(&S.d_full));
    mbar_wait_bounded(smem_u32(&S.d_full), 0);
  } else if (warp >= 2) {
    const int qd = warp & 3;                       // TMEM lane quarter of this warp
    const int f = m0 + qd * 32 + lane;             // this thread's output feature
    bool ok = fw_wait(smem_u32(&S.d_full), 0, abort) && n > 0;
    ok = __all_sync(0xffffffffu, ok) && !*abort;
    tc_fence_after();
    if (J.swiglu_I > 0) {
      // up values (lanes 64-127) through shared memory (the stages are idle now: every
      // copy was consumed by an MMA that has completed) to the gate lanes' threads
      float* up = reinterpret_cast<float*>(sm);    // [Rp][64]
      const uint32_t la = tbase + ((uint32_t)(qd * 32) << 16);
      if (ok && qd >= 2) {
        for (int c0 = 0; c0 < J.Rp; c0 += 16) {
          float v[16];
          tmem_ld16(la + (uint32_t)c0, v);
#pragma unroll
          for (int c = 0; c < 16; ++c) up[(c0 + c) * 64 + (qd - 2) * 32 + lane] = v[c];
        }
      }
      fw_bar(1, 128);
      if (ok && qd < 2) {
        const int fl = qd * 32 + lane;             // gate row within the CTA's 64
        __nv_bfloat16* out = J.A + m0 + fl;
        for (int c0 = 0; c0 < J.Rp; c0 += 16) {
          float v[16];
          tmem_ld16(la + (uint32_t)c0, v);
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            const int r = c0 + c;
            const float g = v[c], u = up[r * 64 + fl];
            const float a = r < J.R ? g / (1.0f + expf(-g)) * u : 0.f;
            out[(int64_t)r * J.swiglu_I] = __float2bfloat16_rn(a);
          }
        }
      }
    } else if (ok) {
      const uint32_t la = tbase + ((uint32_t)(qd * 32) << 16);
      float* out = J.part + (int64_t)split * J.Rp * J.n_out + f;
      for (int c0 = 0; c0 < J.Rp; c0 += 16) {
        float v[16];
        tmem_ld16(la + (uint32_t)c0, v);
#pragma unroll
        for (int c = 0; c < 16; ++c)
          if (c0 + c < J.R) out[(int64_t)(c0 + c) * J.n_out] = v[c];
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && S.abort) atomicOr(J.status, kStatusTimeout);
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tbase, 64);
}

// ===========================================================================
// Element-wise steps
// ===========================================================================
struct NormJob {
  float* H;                    // [R][D]
  const __nv_bfloat16* h_in;   // [R][D] or NULL: H = h_in instead of H += partials
  const float* part;           // [splits][Rp][D] or NULL
  int splits;
  const __nv_bfloat16* w;      // [D] or NULL: no normalisation
  __nv_bfloat16* X;            // [Rp][D] (rows >= R zero)
  float* ssq;                  // [R][chunks] partial sums of squares
  unsigned int* ticket;        // [R] arrival counters (never reset: taken modulo chunks)
  int D, R, Rp, chunks;
  float eps;
};

constexpr int kNormCols = 512;   // columns per CTA (2 per thread)

// Grid (chunks = D / 512, Rp). Each CTA adds the partial sums of its 512 columns of a row
// in split order and writes H; with normalisation it also writes its sum of squares, and
// the CTA that completes the row's count (an atomic ticket) sums the chunks' squares in
// chunk order and writes X = bf16(H * rsqrt * w) for the whole row.
__global__ void __launch_bounds__(256) k_fw_norm(const NormJob J) {
  __shared__ float red[8];
  __shared__ int s_last;
  pdl_wait();
  pdl_release();
  const int r = blockIdx.y, c0 = blockIdx.x * kNormCols, t = threadIdx.x;
  const int D = J.D;
  const int x = c0 + 2 * t;                 // this thread's two columns (D is even)
  const bool in = x < D;
  if (r >= J.R) {
    if (J.w && in)
      reinterpret_cast<__nv_bfloat162*>(J.X + (int64_t)r * D)[x >> 1] = __floats2bfloat162_rn(0.f, 0.f);
    return;
  }
  float2 h = make_float2(0.f, 0.f);
  if (in) {
    if (J.h_in) {
      const __nv_bfloat162 b = reinterpret_cast<const __nv_bfloat162*>(J.h_in + (int64_t)r * D)[x >> 1];
      h = make_float2(__low2float(b), __high2float(b));
    } else {
      h = reinterpret_cast<const float2*>(J.H + (int64_t)r * D)[x >> 1];
    }
    if (J.part) {
      // up to 16 splits' partials loaded together (one memory latency), summed in order
      int s = 0;
      if (J.splits <= 16) {
        float2 v[16];
#pragma unroll
        for (int u = 0; u < 16; ++u)
          if (u < J.splits)
            v[u] = reinterpret_cast<const float2*>(J.part + ((int64_t)u * J.Rp + r) * D)[x >> 1];
#pragma unroll
        for (int u = 0; u < 16; ++u)
          if (u < J.splits) {
            h.x += v[u].x;
            h.y += v[u].y;
          }
        s = J.splits;
      }
      for (; s < J.splits; ++s) {
        const float2 v = reinterpret_cast<const float2*>(J.part + ((int64_t)s * J.Rp + r) * D)[x >> 1];
        h.x += v.x;
        h.y += v.y;
      }
    }
    reinterpret_cast<float2*>(J.H + (int64_t)r * D)[x >> 1] = h;
  }
  if (!J.w) return;
  float ss = fmaf(h.y, h.y, h.x * h.x);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((t & 31) == 0) red[t >> 5] = ss;
  __syncthreads();
  if (t == 0) {
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += red[w];
    J.ssq[(int64_t)r * J.chunks + blockIdx.x] = tot;
    __threadfence();
    const unsigned int old = atomicAdd(J.ticket + r, 1u);
    s_last = (old % (unsigned)J.chunks) == (unsigned)(J.chunks - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  float tot = 0.f;
  for (int c = 0; c < J.chunks; ++c) tot += __ldcg(J.ssq + (int64_t)r * J.chunks + c);
  const float inv = 1.0f / sqrtf(tot / (float)D + J.eps);
  // the row's H and weights loaded together (one memory latency) where D <= 16 x 512
  constexpr int kIt = 16;
  if (D <= kIt * 512) {
    float2 hv[kIt];
    __nv_bfloat162 wv[kIt];
#pragma unroll
    for (int it = 0; it < kIt; ++it) {
      const int y = 2 * t + 512 * it;
      if (y < D) {
        hv[it] = __ldcg(reinterpret_cast<const float2*>(J.H + (int64_t)r * D + y));
        wv[it] = reinterpret_cast<const __nv_bfloat162*>(J.w)[y >> 1];
      }
    }
#pragma unroll
    for (int it = 0; it < kIt; ++it) {
      const int y = 2 * t + 512 * it;
      if (y < D)
        reinterpret_cast<__nv_bfloat162*>(J.X + (int64_t)r * D)[y >> 1] = __floats2bfloat162_rn(
            hv[it].x * inv * __low2float(wv[it]), hv[it].y * inv * __high2float(wv[it]));
    }
    return;
  }
  for (int y = 2 * t; y < D; y += 512) {
    const float2 hv = __ldcg(reinterpret_cast<const float2*>(J.H + (int64_t)r * D + y));
    const __nv_bfloat162 wv = reinterpret_cast<const __nv_bfloat162*>(J.w)[y >> 1];
    reinterpret_cast<__nv_bfloat162*>(J.X + (int64_t)r * D)[y >> 1] =
        __floats2bfloat162_rn(hv.x * inv * __low2float(wv), hv.y * inv * __high2float(wv));
  }
}

// cos and sin of the RoPE angles pos * theta^(-2j/d) of every question row (computed in
// fp64, stored as fp32): [R][64] pairs.
// The same in one pass with one CTA per row (D / 4 threads, four columns each; D <= 4096):
// the row's partials loaded eight splits at a time, its sum of squares reduced in the
// CTA (warps in order), then normalised; no second kernel phase and no arrival counters.
__global__ void __launch_bounds__(1024) k_fw_norm_row(const NormJob J) {
  __shared__ float red[32];
  __shared__ float s_inv;
  pdl_wait();
  pdl_release();
  const int r = blockIdx.x, t = threadIdx.x, D = J.D;
  const int x = 4 * t;
  if (r >= J.R) {
    if (J.w) {
      const __nv_bfloat162 z = __floats2bfloat162_rn(0.f, 0.f);
      reinterpret_cast<__nv_bfloat162*>(J.X + (int64_t)r * D + x)[0] = z;
      reinterpret_cast<__nv_bfloat162*>(J.X + (int64_t)r * D + x)[1] = z;
    }
    return;
  }
  float4 h;
  if (J.h_in) {
    const uint2 b = *reinterpret_cast<const uint2*>(J.h_in + (int64_t)r * D + x);
    h = make_float4(__uint_as_float(b.x << 16), __uint_as_float(b.x & 0xffff0000u),
                    __uint_as_float(b.y << 16), __uint_as_float(b.y & 0xffff0000u));
  } else {
    h = *reinterpret_cast<const float4*>(J.H + (int64_t)r * D + x);
  }
  if (J.part) {
    // eight splits' partials at a time, summed in split order
    for (int s0 = 0; s0 < J.splits; s0 += 8) {
      float4 v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (s0 + u < J.splits)
          v[u] = *reinterpret_cast<const float4*>(J.part + ((int64_t)(s0 + u) * J.Rp + r) * D + x);
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (s0 + u < J.splits) {
          h.x += v[u].x;
          h.y += v[u].y;
          h.z += v[u].z;
          h.w += v[u].w;
        }
    }
  }
  *reinterpret_cast<float4*>(J.H + (int64_t)r * D + x) = h;
  if (!J.w) return;
  float ss = fmaf(h.w, h.w, fmaf(h.z, h.z, fmaf(h.y, h.y, h.x * h.x)));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((t & 31) == 0) red[t >> 5] = ss;
  __syncthreads();
  if (t == 0) {
    float tot = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
    s_inv = 1.0f / sqrtf(tot / (float)D + J.eps);
  }
  __syncthreads();
  const float inv = s_inv;
  const uint2 wb = *reinterpret_cast<const uint2*>(J.w + x);
  const float w0 = __uint_as_float(wb.x << 16), w1 = __uint_as_float(wb.x & 0xffff0000u);
  const float w2 = __uint_as_float(wb.y << 16), w3 = __uint_as_float(wb.y & 0xffff0000u);
  __nv_bfloat162* dst = reinterpret_cast<__nv_bfloat162*>(J.X + (int64_t)r * D + x);
  dst[0] = __floats2bfloat162_rn(h.x * inv * w0, h.y * inv * w1);
  dst[1] = __floats2bfloat162_rn(h.z * inv * w2, h.w * inv * w3);
}

__global__ void __launch_bounds__(64) k_fw_rope(float2* tab, int64_t pos0, double theta) {
  const int r = blockIdx.x, j = threadIdx.x;
  pdl_wait();     // (an earlier forward's kernels may still read the table)
  pdl_release();
  const double inv = pow(theta, -2.0 * (double)j / (double)kHeadDim);
  double sd, cd;
  sincos((double)(pos0 + r) * inv, &sd, &cd);
  tab[r * 64 + j] = make_float2((float)cd, (float)sd);
}

struct QkvJob {
  const float* part;           // [splits][Rp][(Hq + 2 Hkv) d]
  int splits, Rp, R;
  const __nv_bfloat16* bias;   // [(Hq + 2 Hkv) d] or NULL
  int Hq, Hkv;
  const float2* rope;          // [R][64] (cos, sin)
  __nv_bfloat16* q;            // [R][Hq][d] (the caller's Q^i)
  __nv_bfloat16* k;            // [R][Hkv][d]
  __nv_bfloat16* v;            // [R][Hkv][d]
};

// Grid (R, Hq + 2 Hkv); thread j < 64 owns the pair (j, j + 64) of one head.
__global__ void __launch_bounds__(64) k_fw_qkv(const QkvJob J) {
  const int r = blockIdx.x, t = blockIdx.y, j = threadIdx.x;
  pdl_wait();
  pdl_release();
  const int n_out = (J.Hq + 2 * J.Hkv) * kHeadDim;
  const int f0 = t * kHeadDim + j, f1 = f0 + 64;
  float y0 = 0.f, y1 = 0.f;
  int s = 0;
  if (J.splits <= 16) {
    // every split's partial loaded together (one memory latency), summed in order
    float a[16], b[16];
#pragma unroll
    for (int u = 0; u < 16; ++u)
      if (u < J.splits) {
        const float* p = J.part + ((int64_t)u * J.Rp + r) * n_out;
        a[u] = p[f0];
        b[u] = p[f1];
      }
#pragma unroll
    for (int u = 0; u < 16; ++u)
      if (u < J.splits) {
        y0 += a[u];
        y1 += b[u];
      }
    s = J.splits;
  }
  for (; s < J.splits; ++s) {
    const float* p = J.part + ((int64_t)s * J.Rp + r) * n_out;
    y0 += p[f0];
    y1 += p[f1];
  }
  if (J.bias) {
    y0 += __bfloat162float(J.bias[f0]);
    y1 += __bfloat162float(J.bias[f1]);
  }
  __nv_bfloat16* dst;
  if (t < J.Hq + J.Hkv) {
    const float2 cs = J.rope[r * 64 + j];
    const float a = fmaf(y0, cs.x, -y1 * cs.y);
    const float b = fmaf(y1, cs.x, y0 * cs.y);
    y0 = a;
    y1 = b;
    dst = t < J.Hq ? J.q + ((int64_t)r * J.Hq + t) * kHeadDim
                   : J.k + ((int64_t)r * J.Hkv + (t - J.Hq)) * kHeadDim;
  } else {
    dst = J.v + ((int64_t)r * J.Hkv + (t - J.Hq - J.Hkv)) * kHeadDim;
  }
  dst[j] = __float2bfloat16_rn(y0);
  dst[j + 64] = __float2bfloat16_rn(y1);
}

struct SwigluJob {
  const float* part;           // [splits][Rp][2 I]
  int splits, Rp, R, I;
  __nv_bfloat16* A;            // [Rp][I]
};

__global__ void __launch_bounds__(256) k_fw_swiglu(const SwigluJob J) {
  const int64_t x = (int64_t)blockIdx.x * 256 + threadIdx.x;
  pdl_wait();
  pdl_release();
  if (x >= (int64_t)J.Rp * J.I) return;
  const int r = (int)(x / J.I), f = (int)(x - (int64_t)r * J.I);
  float a = 0.f;
  if (r < J.R) {
    float g = 0.f, u = 0.f;
    for (int s = 0; s < J.splits; ++s) {
      const float* p = J.part + ((int64_t)s * J.Rp + r) * (2 * J.I);
      g += p[f];
      u += p[J.I + f];
    }
    a = g / (1.0f + expf(-g)) * u;
  }
  J.A[x] = __float2bfloat16_rn(a);
}

// ===========================================================================
// Attention of the question rows over the layer's stored tokens
// ===========================================================================
constexpr int kAtThreads = 192;            // warp 0 TMA, warp 1 MMA, warps 2-5 rows
constexpr int kAtTile = 64;                // tokens per tile
constexpr int kAtTileBytes = kAtTile * kHeadDim * 2;   // 16 KB of keys or values
constexpr int kAtQBytes = 128 * kHeadDim * 2;          // 32 KB: 128 rows x 128 dims
constexpr float kAtLazy = 8.0f;            // raise the running max only past this margin

struct AttnJob {
  int layer;
  int Hq, Hkv, G, R, Rp, GRp, halves;
  int n_tok;                       // stored tokens of every slab
  int chunks;
  const __nv_bfloat16* q;          // [R][Hq][d] this layer's question rows
  float* opart;                    // [Hkv][chunks][halves * 128][d] unnormalised O
  float2* mlpart;                  // [Hkv][chunks][halves * 128] (m, l)
  uint32_t* status;
};

// Barriers, at the end of the dynamic shared memory (no static shared memory, so the
// dynamic region starts on the 1024-byte boundary the swizzled tiles need).
struct AtBars {
  unsigned long long kfull[2], kempty[2], vfull[2], vempty[2], sfull[2];
  unsigned long long pfull, pvdone, q_ready, final_mma;
  uint32_t taddr;
  int abort;
};

constexpr int kAtSmem = kAtQBytes + 4 * kAtTileBytes + (int)sizeof(AtBars);

// grid (chunks, halves, Hkv), two CTAs per SM (256 TMEM columns, ~113 KB of shared memory
// each). Rows rho = h * Rp + r (h < G) of key head g; this CTA takes rho in
// [128 * half, 128 * half + 128), one thread per row (TMEM lane). Per tile j of 64 tokens:
//   TMA    K(j), V(j) into two-stage rings
//   MMA    S(j) = Q K(j)^T into one of two TMEM buffers (64 columns) as soon as K(j) is in
//          and O += P(j - 2) V(j - 2) has been issued; O += P(j) V(j) once P(j) is written,
//          its A operand read from TMEM (event loop)
//   rows   S(j) -> m, P(j) = bf16(2^(s - m)) back into the first 32 columns of S(j)'s
//          buffer (two weights per column), l; the running maximum raised only past 8
//          (log2), then O and l rescaled in TMEM
// P never passes through shared memory: the tensor cores' operand reads there are only Q,
// K and V (with the TMA writes of K and V, shared-memory bandwidth is this kernel's bound).
// The second CTA on the SM fills the gaps of each CTA's chain of dependent steps.
__global__ void __launch_bounds__(256, 2)
    k_fw_attn(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
              const AttnJob J) {
  extern __shared__ __align__(1024) unsigned char sm[];
  unsigned char* qs = sm;                        // A operand of S = Q K^T: 128 rows x 128 dims
  unsigned char* kr = qs + kAtQBytes;            // 2 key stages
  unsigned char* vr = kr + 2 * kAtTileBytes;     // 2 value stages
  AtBars& S = *reinterpret_cast<AtBars*>(vr + 2 * kAtTileBytes);
  const int chunk = blockIdx.x, half = blockIdx.y, g = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if ((smem_u32(sm) & 1023u) != 0u) {             // the swizzled tiles need the boundary
    if (threadIdx.x == 0) atomicOr(J.status, kStatusInternal);
    return;
  }
  const int T = (J.n_tok + kAtTile - 1) / kAtTile;
  const int t0 = (int)((int64_t)T * chunk / J.chunks);
  const int t1 = (int)((int64_t)T * (chunk + 1) / J.chunks);
  const int n = t1 - t0;
  volatile int* abort = &S.abort;
  if (threadIdx.x == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(smem_u32(&S.kfull[b]), 1);
      mbar_init(smem_u32(&S.kempty[b]), 1);
      mbar_init(smem_u32(&S.vfull[b]), 1);
      mbar_init(smem_u32(&S.vempty[b]), 1);
      mbar_init(smem_u32(&S.sfull[b]), 1);
    }
    mbar_init(smem_u32(&S.pfull), 128);
    mbar_init(smem_u32(&S.pvdone), 1);
    mbar_init(smem_u32(&S.q_ready), 1);
    mbar_init(smem_u32(&S.final_mma), 1);
    S.abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&S.taddr), 256);   // S in columns 0-127 (two buffers), O at 128
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_release();
  const uint32_t tbase = S.taddr;
  // tensor maps [P][Hkv][n_tok][d]: a tile past the stored tokens reads zeros
  const int y0 = t0 * kAtTile;
  if (warp == 0 && lane == 0) {
    // ---- TMA producer: K(j) and V(j) into their rings ----
    tma_prefetch_map(&kmap);
    tma_prefetch_map(&vmap);
    int klast[2] = {-1, -1}, vlast[2] = {-1, -1};
    for (int j = 0; j < n && !*abort; ++j) {
      const int st = j & 1;
      const int y = y0 + j * kAtTile;
      if (j >= 2 && !fw_wait(smem_u32(&S.kempty[st]), ((j >> 1) - 1) & 1, abort)) break;
      uint32_t bar = smem_u32(&S.kfull[st]);
      uint32_t dst = smem_u32(kr + st * kAtTileBytes);
      mbar_expect_tx(bar, kAtTileBytes);
      tma_load_4d(dst, &kmap, bar, 0, y, g, J.layer);
      tma_load_4d(dst + kAtTileBytes / 2, &kmap, bar, 64, y, g, J.layer);
      klast[st] = j;
      if (j >= 2 && !fw_wait(smem_u32(&S.vempty[st]), ((j >> 1) - 1) & 1, abort)) break;
      bar = smem_u32(&S.vfull[st]);
      dst = smem_u32(vr + st * kAtTileBytes);
      mbar_expect_tx(bar, kAtTileBytes);
      tma_load_4d(dst, &vmap, bar, 0, y, g, J.layer);
      tma_load_4d(dst + kAtTileBytes / 2, &vmap, bar, 64, y, g, J.layer);
      vlast[st] = j;
    }
    for (int b = 0; b < 2; ++b) {
      if (klast[b] >= 0) mbar_wait_bounded(smem_u32(&S.kfull[b]), (klast[b] >> 1) & 1);
      if (vlast[b] >= 0) mbar_wait_bounded(smem_u32(&S.vfull[b]), (vlast[b] >> 1) & 1);
    }
  } else if (warp == 1 && lane == 0) {
    // ---- MMA issuer, an event loop over two queues: S(j1) = Q K(j1)^T as soon as its
    // keys are in and O += P(j1 - 2) V(j1 - 2) (the last reader of its TMEM buffer) has
    // been issued (the MMAs of one thread run in issue order), O += P(j2) V(j2) as soon as
    // its weights are written (non-blocking tests, so neither queue holds back the other) ----
    const uint32_t id1 = idesc_bf16_f32(128, kAtTile, false, false);
    const uint32_t id2 = idesc_bf16_f32(128, 128, false, true);
    const uint32_t qa = smem_u32(qs);
    if (fw_wait(smem_u32(&S.q_ready), 0, abort)) {
      int j1 = 0, j2 = 0;
      uint64_t t_idle = 0;
      uint32_t idle = 0;
      while (j2 < n) {
        bool did = false;
        if (j1 < n) {
          const int st = j1 & 1;
          const bool ready =
              j2 >= j1 - 1 && mbar_test_wait(smem_u32(&S.kfull[st]), (j1 >> 1) & 1);
          if (ready) {
            tc_fence_after();
            const uint32_t ka = smem_u32(kr + st * kAtTileBytes);
            const uint32_t d = tbase + (uint32_t)st * 64u;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              // Q: two 64-dim halves 16 KB apart; K tile: two 64-dim halves 8 KB apart
              const uint32_t qo = (k >> 2) * 16384 + (k & 3) * 32;
              const uint32_t ko = (k >> 2) * (kAtTileBytes / 2) + (k & 3) * 32;
              umma_bf16(d, sdesc_sw128(qa + qo, 16, 1024), sdesc_sw128(ka + ko, 16, 1024), id1,
                        k > 0 ? 1u : 0u);
            }
            umma_commit(smem_u32(&S.sfull[st]));
            umma_commit(smem_u32(&S.kempty[st]));
            ++j1;
            did = true;
          }
        }
        if (j2 < j1) {
          const int st = j2 & 1;
          if (mbar_test_wait(smem_u32(&S.pfull), j2 & 1) &&
              mbar_test_wait(smem_u32(&S.vfull[st]), (j2 >> 1) & 1)) {
            tc_fence_after();
            const uint32_t va = smem_u32(vr + st * kAtTileBytes);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              // P: in TMEM, 16 tokens = 8 columns per K step; V: N = dims MN-major (two
              // 64-dim blocks 8 KB apart), 16 tokens = 2048 bytes per K step
              umma_bf16_ts(tbase + 128u, tbase + (uint32_t)(st * 64 + k * 8),
                           sdesc_sw128(va + k * 2048, kAtTileBytes / 2, 1024), id2,
                           (j2 > 0 || k > 0) ? 1u : 0u);
            }
            umma_commit(smem_u32(&S.vempty[st]));
            umma_commit(smem_u32(&S.pvdone));
            ++j2;
            did = true;
          }
        }
        if (did) {
          idle = 0;
        } else if (__nanosleep(32), (++idle & 255u) == 0u) {
          // bounded: give up after ~1 s without progress, or when another role did
          const uint64_t now = global_ns();
          if (idle == 256u) t_idle = now;
          if (*abort || now - t_idle > 1000000000ull || idle >= kDefaultWaitPolls) {
            *abort = 1;
            break;
          }
        }
      }
    }
    umma_commit(smem_u32(&S.final_mma));
    mbar_wait_bounded(smem_u32(&S.final_mma), 0);
  } else if (warp >= 2) {
    // ---- rows: one per thread (TMEM lane) ----
    const int e = threadIdx.x - 64;
    const int qd = warp & 3;
    const int rl = qd * 32 + lane;                 // row within the CTA's 128
    const int rho = half * 128 + rl;
    const int hl = rho / J.Rp, r = rho - hl * J.Rp;
    const bool valid = hl < J.G && r < J.R;
    // (the keys and values stream in meanwhile: they do not depend on the previous kernel)
    pdl_wait();
    // question rows -> 128-byte swizzled K-major tile (two halves of 64 dims); a thread's
    // 16 chunks loaded together, then stored (one memory latency)
    {
      uint4 v[16];
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const int x = e + 128 * u;
        const int row = x >> 4, c = x & 15;
        const int rr = half * 128 + row;
        const int h2 = rr / J.Rp, r2 = rr - h2 * J.Rp;
        v[u] = make_uint4(0u, 0u, 0u, 0u);
        if (h2 < J.G && r2 < J.R)
          v[u] = *reinterpret_cast<const uint4*>(J.q + ((int64_t)r2 * J.Hq + g * J.G + h2) *
                                                           kHeadDim + 8 * c);
      }
#pragma unroll
      for (int u = 0; u < 16; ++u) {
        const int x = e + 128 * u;
        const int row = x >> 4, c = x & 15;
        *reinterpret_cast<uint4*>(qs + (c >> 3) * 16384 + row * 128 + (((c & 7) ^ (row & 7)) << 4)) =
            v[u];
      }
    }
    fence_proxy_async_smem();
    fw_bar(1, 128);
    if (e == 0) mbar_arrive(smem_u32(&S.q_ready));
    const uint32_t la = tbase + ((uint32_t)(qd * 32) << 16);
    const unsigned long long sc2 = f2pack(kScoreScale, kScoreScale);
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < n; ++j) {
      const int st = j & 1;
      ok = ok && fw_wait(smem_u32(&S.sfull[st]), (j >> 1) & 1, abort);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      float s[64];
      tmem_ld32x2(la + st * 64u, la + st * 64u + 32u, *reinterpret_cast<float(*)[32]>(s),
                  *reinterpret_cast<float(*)[32]>(s + 32));
      const int nv = min(kAtTile, J.n_tok - (t0 + j) * kAtTile);   // valid tokens
      if (nv < kAtTile) {
#pragma unroll
        for (int c = 0; c < kAtTile; ++c)
          if (c >= nv) s[c] = -INFINITY;
      }
      float a0 = -INFINITY, a1 = -INFINITY;
#pragma unroll
      for (int c = 0; c < kAtTile; c += 4) {
        a0 = fmax3(a0, s[c], s[c + 1]);
        a1 = fmax3(a1, s[c + 2], s[c + 3]);
      }
      const float mt = fmaxf(a0, a1) * kScoreScale;
      const bool raise = mt > m + kAtLazy;
      const float m_new = raise ? mt : m;
      // P = 2^(s - m_new) rounded to bf16 for the tensor cores; the scaling and l (the sum
      // of the weights before rounding) on packed pairs
      uint32_t pk[32];
      const unsigned long long nm2 = f2pack(-m_new, -m_new);
      unsigned long long acc0 = 0ull, acc1 = 0ull;
#pragma unroll
      for (int c = 0; c < 32; ++c) {
        const unsigned long long x = ffma2(f2pack(s[2 * c], s[2 * c + 1]), sc2, nm2);
        const float p0 = fast_exp2(f2lo(x)), p1 = fast_exp2(f2hi(x));
        const __nv_bfloat162 b2 = __floats2bfloat162_rn(p0, p1);
        pk[c] = *reinterpret_cast<const uint32_t*>(&b2);
        if (c & 1) acc1 = fadd2(acc1, f2pack(p0, p1));
        else acc0 = fadd2(acc0, f2pack(p0, p1));
      }
      // P(j) over S(j) in TMEM (O += P(j - 2) V(j - 2), the buffer's last reader, completed
      // before S(j) was computed)
      tmem_st32u(la + st * 64u, pk);
      // O is free once O += P(j - 1) V(j - 1) has completed; a raised maximum then rescales
      // O (and l) before P(j) is released
      if (j >= 1) {
        ok = fw_wait(smem_u32(&S.pvdone), (j - 1) & 1, abort);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) break;
        tc_fence_after();
        if (__any_sync(0xffffffffu, raise)) {
          const float fac = raise ? fast_exp2(m - m_new) : 1.0f;
#pragma unroll 1
          for (int c0 = 0; c0 < 128; c0 += 32) {
            float o[32];
            tmem_ld32(la + 128u + (uint32_t)c0, o);
#pragma unroll
            for (int c = 0; c < 32; ++c) o[c] *= fac;
            tmem_st32(la + 128u + (uint32_t)c0, o);
          }
          l *= fac;
        }
      }
      m = m_new;
      l += (f2lo(acc0) + f2hi(acc0)) + (f2lo(acc1) + f2hi(acc1));
      tc_fence_before();
      mbar_arrive(smem_u32(&S.pfull));
    }
    if (ok && n > 0) {
      ok = fw_wait(smem_u32(&S.pvdone), (n - 1) & 1, abort);
      ok = __all_sync(0xffffffffu, ok);
    }
    tc_fence_after();
    const int64_t prow_out = ((int64_t)g * J.chunks + chunk) * (J.halves * 128) + rho;
    if (ok && !*abort) {
      for (int c0 = 0; c0 < 128; c0 += 32) {
        float o[32];
        tmem_ld32(la + 128u + (uint32_t)c0, o);
        if (valid && n > 0) {
          float4* dst = reinterpret_cast<float4*>(J.opart + prow_out * kHeadDim + c0);
#pragma unroll
          for (int c = 0; c < 8; ++c) dst[c] = make_float4(o[4 * c], o[4 * c + 1], o[4 * c + 2], o[4 * c + 3]);
        }
      }
      if (valid) J.mlpart[prow_out] = n > 0 ? make_float2(m, l) : make_float2(-INFINITY, 0.f);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && S.abort) atomicOr(J.status, kStatusTimeout);
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tbase, 256);
}

struct AttnOutJob {
  int Hq, Hkv, G, R, Rp, halves, chunks;
  const __nv_bfloat16* q;          // [R][Hq][d]
  const __nv_bfloat16* k;          // [R][Hkv][d] the question's own keys
  const __nv_bfloat16* v;          // [R][Hkv][d]
  const float* opart;
  const float2* mlpart;
  __nv_bfloat16* o;                // [Rp][Hq d] (rows >= R zero)
  const uint32_t* status;
};

// One CTA per (row r of Rp, query head h), eight warps. The row's items are the chunks'
// partials (m, l, O) and its own rows 0..r (score s, weight 1, value v); warp w takes
// chunks w, w + 8, ... and own rows w, w + 8, ..., loads them together, and reduces them
// under its own maximum in item order (lane: dims 4 lane .. 4 lane + 3). The eight warps'
// results are then merged in warp order under the common maximum.
__global__ void __launch_bounds__(256) k_fw_attn_out(const AttnOutJob J) {
  __shared__ float4 s_acc[8][32];
  __shared__ float s_m[8], s_l[8];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x / J.Hq, h = blockIdx.x - r * J.Hq;
  pdl_wait();
  pdl_release();
  __nv_bfloat16* dst = J.o + (int64_t)r * J.Hq * kHeadDim + h * kHeadDim + 4 * lane;
  if (r >= J.R || (*(volatile const uint32_t*)J.status & kStatusTimeout)) {
    if (warp == 0) {
      const __nv_bfloat162 z = __floats2bfloat162_rn(0.f, 0.f);
      reinterpret_cast<__nv_bfloat162*>(dst)[0] = z;
      reinterpret_cast<__nv_bfloat162*>(dst)[1] = z;
    }
    return;
  }
  const int g = h / J.G, hl = h - g * J.G;
  const int rho = hl * J.Rp + r;
  const int rows = J.halves * 128;
  constexpr int kC = 8;                         // chunks per warp loaded together (38 / 8 = 5)
  constexpr int kO = 8;                         // own rows per warp (R <= 64)
  // own rows jr = warp + 8 u: scores (one dot per row, lanes summed in a fixed butterfly)
  const uint2 qv = *reinterpret_cast<const uint2*>(J.q + ((int64_t)r * J.Hq + h) * kHeadDim + 4 * lane);
  const float q0 = __uint_as_float(qv.x << 16), q1 = __uint_as_float(qv.x & 0xffff0000u);
  const float q2 = __uint_as_float(qv.y << 16), q3 = __uint_as_float(qv.y & 0xffff0000u);
  float so[kO];
  uint2 vo[kO];
#pragma unroll
  for (int u = 0; u < kO; ++u) {
    const int jr = warp + 8 * u;
    so[u] = -INFINITY;
    vo[u] = make_uint2(0u, 0u);
    if (jr <= r) {
      const uint2 kv = *reinterpret_cast<const uint2*>(J.k + ((int64_t)jr * J.Hkv + g) * kHeadDim + 4 * lane);
      vo[u] = *reinterpret_cast<const uint2*>(J.v + ((int64_t)jr * J.Hkv + g) * kHeadDim + 4 * lane);
      float d = q0 * __uint_as_float(kv.x << 16);
      d = fmaf(q1, __uint_as_float(kv.x & 0xffff0000u), d);
      d = fmaf(q2, __uint_as_float(kv.y << 16), d);
      d = fmaf(q3, __uint_as_float(kv.y & 0xffff0000u), d);
      so[u] = d;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
#pragma unroll
    for (int u = 0; u < kO; ++u) so[u] += __shfl_xor_sync(0xffffffffu, so[u], o);
#pragma unroll
  for (int u = 0; u < kO; ++u) so[u] = warp + 8 * u <= r ? so[u] * kScoreScale : -INFINITY;
  // this warp's chunks c = warp + 8 u
  float M = -INFINITY;
#pragma unroll
  for (int u = 0; u < kO; ++u) M = fmaxf(M, so[u]);
  float L = 0.f;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int c0 = warp; c0 < J.chunks; c0 += 8 * kC) {
    float2 ml[kC];
    float4 ov[kC];
#pragma unroll
    for (int u = 0; u < kC; ++u) {
      const int c = c0 + 8 * u;
      ml[u] = make_float2(-INFINITY, 0.f);
      if (c < J.chunks) {
        const int64_t pr = ((int64_t)g * J.chunks + c) * rows + rho;
        ml[u] = J.mlpart[pr];
        ov[u] = reinterpret_cast<const float4*>(J.opart + pr * kHeadDim)[lane];
      }
    }
    float Mb = M;
#pragma unroll
    for (int u = 0; u < kC; ++u)
      if (ml[u].y > 0.f) Mb = fmaxf(Mb, ml[u].x);
    if (Mb > M) {                               // the batch raised the warp's maximum
      const float f = M == -INFINITY ? 0.f : fast_exp2(M - Mb);
      L *= f;
      acc.x *= f;
      acc.y *= f;
      acc.z *= f;
      acc.w *= f;
      M = Mb;
    }
#pragma unroll
    for (int u = 0; u < kC; ++u) {
      if (!(ml[u].y > 0.f)) continue;
      const float wgt = fast_exp2(ml[u].x - M);
      L = fmaf(ml[u].y, wgt, L);
      acc.x = fmaf(ov[u].x, wgt, acc.x);
      acc.y = fmaf(ov[u].y, wgt, acc.y);
      acc.z = fmaf(ov[u].z, wgt, acc.z);
      acc.w = fmaf(ov[u].w, wgt, acc.w);
    }
  }
#pragma unroll
  for (int u = 0; u < kO; ++u) {
    if (warp + 8 * u > r) break;
    const float wgt = fast_exp2(so[u] - M);
    L += wgt;
    acc.x = fmaf(__uint_as_float(vo[u].x << 16), wgt, acc.x);
    acc.y = fmaf(__uint_as_float(vo[u].x & 0xffff0000u), wgt, acc.y);
    acc.z = fmaf(__uint_as_float(vo[u].y << 16), wgt, acc.z);
    acc.w = fmaf(__uint_as_float(vo[u].y & 0xffff0000u), wgt, acc.w);
  }
  s_acc[warp][lane] = acc;
  if (lane == 0) {
    s_m[warp] = M;
    s_l[warp] = L;
  }
  __syncthreads();
  if (warp != 0) return;
  float Mt = -INFINITY;
#pragma unroll
  for (int w = 0; w < 8; ++w) Mt = fmaxf(Mt, s_m[w]);
  float Lt = 0.f;
  float4 at = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int w = 0; w < 8; ++w) {
    if (s_m[w] == -INFINITY) continue;
    const float f = fast_exp2(s_m[w] - Mt);
    const float4 a = s_acc[w][lane];
    Lt = fmaf(s_l[w], f, Lt);
    at.x = fmaf(a.x, f, at.x);
    at.y = fmaf(a.y, f, at.y);
    at.z = fmaf(a.z, f, at.z);
    at.w = fmaf(a.w, f, at.w);
  }
  const float inv = 1.0f / Lt;
  reinterpret_cast<__nv_bfloat162*>(dst)[0] = __floats2bfloat162_rn(at.x * inv, at.y * inv);
  reinterpret_cast<__nv_bfloat162*>(dst)[1] = __floats2bfloat162_rn(at.z * inv, at.w * inv);
}

// ===========================================================================
// Host: one forward
// ===========================================================================
namespace {

int gemm_stages(int Rp) {
  const int stage = kGmABytes + Rp * 128;
  int s = (110 * 1024) / stage;              // two CTAs per SM
  return s < 2 ? 2 : (s > kGmMaxStages ? kGmMaxStages : s);
}

// K splits per output tile: as many as keep the grid within one wave of two CTAs per SM
// (a grid just past the wave leaves a few CTAs running alone at its end)
int gemm_splits(int n_out, int kblocks, int sm_count) {
  const int tiles = n_out / 128;
  int s = (2 * sm_count) / tiles;
  if (s < 1) s = 1;
  if (s > kblocks) s = kblocks;
  if (s > 16) s = 16;
  return s;
}

struct Seg {
  size_t off = 0;
  template <typename T>
  size_t take(size_t count) {
    const size_t o = off;
    off = (off + count * sizeof(T) + 255) & ~(size_t)255;
    return o;
  }
};

struct FwLayout {
  size_t H, X, A, part, k, v, opart, ml, rope, ssq, ticket, total;
  int Rp, halves, chunks, nchunks, sp_qkv, sp_o, sp_gu, sp_d;
};

FwLayout fw_layout(const FwShape& F) {
  FwLayout L{};
  const int D = F.Hq * kHeadDim;
  L.Rp = (F.R + 15) & ~15;
  const int G = F.Hq / F.Hkv;
  L.halves = (G * L.Rp + 127) / 128;
  const int T = (F.n_tok + kAtTile - 1) / kAtTile;
  int c = 2 * F.sm_count / (L.halves * F.Hkv);   // two attention CTAs per SM
  c = c < 1 ? 1 : c;
  L.chunks = T < 1 ? 1 : (T < c ? T : c);
  const int nqkv = (F.Hq + 2 * F.Hkv) * kHeadDim;
  L.sp_qkv = gemm_splits(nqkv, D / 64, F.sm_count);
  L.sp_o = gemm_splits(D, D / 64, F.sm_count);
  L.sp_gu = gemm_splits(2 * F.I, D / 64, F.sm_count);
  L.sp_d = gemm_splits(D, F.I / 64, F.sm_count);
  size_t part = (size_t)L.sp_qkv * nqkv;
  part = std::max(part, (size_t)L.sp_o * D);
  part = std::max(part, (size_t)L.sp_gu * 2 * F.I);
  part = std::max(part, (size_t)L.sp_d * D);
  Seg s;
  L.H = s.take<float>((size_t)F.R * D);
  L.X = s.take<__nv_bfloat16>((size_t)L.Rp * D);
  L.A = s.take<__nv_bfloat16>((size_t)L.Rp * F.I);
  L.part = s.take<float>(part * L.Rp);
  L.k = s.take<__nv_bfloat16>((size_t)F.R * F.Hkv * kHeadDim);
  L.v = s.take<__nv_bfloat16>((size_t)F.R * F.Hkv * kHeadDim);
  L.opart = s.take<float>((size_t)F.Hkv * L.chunks * L.halves * 128 * kHeadDim);
  L.ml = s.take<float2>((size_t)F.Hkv * L.chunks * L.halves * 128);
  L.rope = s.take<float2>((size_t)F.R * 64);
  L.nchunks = (D + kNormCols - 1) / kNormCols;
  L.ssq = s.take<float>((size_t)F.R * L.nchunks);
  L.ticket = s.take<uint32_t>((size_t)F.R + 1);   // the row tickets, then the status word
  L.total = s.off;
  return L;
}

cudaError_t gemm(const void* W, int n_out, int K, const __nv_bfloat16* X, int R, int Rp,
                 int splits, float* part, uint32_t* status, cudaStream_t st, int swiglu_I = 0,
                 __nv_bfloat16* A = nullptr) {
  CUtensorMap wm, xm;
  const uint64_t wd[2] = {(uint64_t)K, (uint64_t)n_out}, ws[1] = {(uint64_t)K * 2};
  const uint32_t wb[2] = {64, swiglu_I > 0 ? 64u : 128u};
  cudaError_t e = encode_bf16_map(&wm, W, 2, wd, ws, wb);
  if (e != cudaSuccess) return e;
  const uint64_t xd[2] = {(uint64_t)K, (uint64_t)Rp}, xs[1] = {(uint64_t)K * 2};
  const uint32_t xb[2] = {64, (uint32_t)Rp};
  e = encode_bf16_map(&xm, X, 2, xd, xs, xb);
  if (e != cudaSuccess) return e;
  GemmJob J;
  J.part = part;
  J.n_out = n_out;
  J.swiglu_I = swiglu_I;
  J.A = A;
  J.R = R;
  J.Rp = Rp;
  J.kblocks = K / 64;
  J.splits = splits;
  J.stages = gemm_stages(Rp);
  J.status = status;
  const int smem = J.stages * (kGmABytes + Rp * 128) + 1024;
  e = ensure_smem((const void*)k_fw_gemm, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_fw_gemm, dim3(swiglu_I > 0 ? swiglu_I / 64 : n_out / 128, splits),
                    dim3(kGmThreads), smem, st, wm, xm, J);
}

}  // namespace

bool forward_supported(int R, int Hq, int Hkv) {
  const int Rp = (R + 15) & ~15;
  return R >= 1 && R <= 64 && (Hq / Hkv) * Rp <= 256;
}

size_t forward_workspace_bytes(const FwShape& F) { return fw_layout(F).total; }

cudaError_t launch_forward(const FwShape& F, const FwArgs& A, cudaStream_t st) {
  const FwLayout L = fw_layout(F);
  unsigned char* ws = static_cast<unsigned char*>(A.workspace);
  float* H = reinterpret_cast<float*>(ws + L.H);
  __nv_bfloat16* X = reinterpret_cast<__nv_bfloat16*>(ws + L.X);
  __nv_bfloat16* Ab = reinterpret_cast<__nv_bfloat16*>(ws + L.A);
  float* part = reinterpret_cast<float*>(ws + L.part);
  __nv_bfloat16* kown = reinterpret_cast<__nv_bfloat16*>(ws + L.k);
  __nv_bfloat16* vown = reinterpret_cast<__nv_bfloat16*>(ws + L.v);
  float* opart = reinterpret_cast<float*>(ws + L.opart);
  float2* ml = reinterpret_cast<float2*>(ws + L.ml);
  float2* rope = reinterpret_cast<float2*>(ws + L.rope);
  float* ssq = reinterpret_cast<float*>(ws + L.ssq);
  unsigned int* ticket = reinterpret_cast<unsigned int*>(ws + L.ticket);
  uint32_t* status = A.status ? A.status : reinterpret_cast<uint32_t*>(ticket + F.R);
  const int D = F.Hq * kHeadDim, G = F.Hq / F.Hkv;
  const int nqkv = (F.Hq + 2 * F.Hkv) * kHeadDim;
  cudaError_t e = cudaMemsetAsync(ticket, 0, (size_t)(F.R + 1) * sizeof(uint32_t), st);
  if (e != cudaSuccess) return e;
  if (A.status && (e = cudaMemsetAsync(status, 0, sizeof(uint32_t), st)) != cudaSuccess) return e;
  if ((e = launch_pdl(k_fw_rope, dim3(F.R), dim3(64), 0, st, rope, F.pos0, F.theta)) != cudaSuccess) return e;
  // stored keys and values of every layer as [P][Hkv][n_tok][d] (the stored tokens of a
  // slab only, so the last tile's rows past them read zeros), tiles of 128 tokens
  CUtensorMap km, vm;
  const uint64_t dims[4] = {(uint64_t)kHeadDim, (uint64_t)F.n_tok, (uint64_t)F.Hkv, (uint64_t)F.P};
  const uint64_t strides[3] = {(uint64_t)kHeadDim * 2, (uint64_t)F.ncap * kHeadDim * 2,
                               (uint64_t)F.Hkv * F.ncap * kHeadDim * 2};
  const uint32_t box[4] = {64, (uint32_t)kAtTile, 1, 1};
  if (F.n_tok > 0) {
    e = encode_bf16_map(&km, F.keys, 4, dims, strides, box);
    if (e != cudaSuccess) return e;
    e = encode_bf16_map(&vm, F.values, 4, dims, strides, box);
    if (e != cudaSuccess) return e;
    e = ensure_smem((const void*)k_fw_attn, kAtSmem);
    if (e != cudaSuccess) return e;
  }
  NormJob nj{};
  nj.H = H;
  nj.D = D;
  nj.R = F.R;
  nj.Rp = L.Rp;
  nj.eps = F.eps;
  nj.ssq = ssq;
  nj.ticket = ticket;
  nj.chunks = L.nchunks;
  const dim3 ngrid(L.nchunks, L.Rp);
  // one CTA per row where a row fits one CTA (four columns per thread), else column chunks
  const bool row_norm = D % 128 == 0 && D / 4 <= 1024;
  auto norm = [&](const NormJob& J) {
    return row_norm ? launch_pdl(k_fw_norm_row, dim3(L.Rp), dim3(D / 4), 0, st, J)
                    : launch_pdl(k_fw_norm, ngrid, dim3(256), 0, st, J);
  };
  for (int i = 0; i < F.P; ++i) {
    const FwLayerW& W = A.layers[i];
    __nv_bfloat16* q = static_cast<__nv_bfloat16*>(A.q_out) + (int64_t)i * F.R * F.Hq * kHeadDim;
    // X = bf16(RMSNorm(H) * ln1); layer 0 starts from the question's rows, later layers
    // add the previous layer's down-projection partials first
    nj.h_in = i == 0 ? static_cast<const __nv_bfloat16*>(A.h_in) : nullptr;
    nj.part = i == 0 ? nullptr : part;
    nj.splits = L.sp_d;
    nj.w = static_cast<const __nv_bfloat16*>(W.ln1);
    nj.X = X;
    if ((e = norm(nj)) != cudaSuccess) return e;
    if ((e = gemm(W.wqkv, nqkv, D, X, F.R, L.Rp, L.sp_qkv, part, status, st)) != cudaSuccess) return e;
    QkvJob qj;
    qj.part = part;
    qj.splits = L.sp_qkv;
    qj.Rp = L.Rp;
    qj.R = F.R;
    qj.bias = static_cast<const __nv_bfloat16*>(W.bqkv);
    qj.Hq = F.Hq;
    qj.Hkv = F.Hkv;
    qj.rope = rope;
    qj.q = q;
    qj.k = kown;
    qj.v = vown;
    if ((e = launch_pdl(k_fw_qkv, dim3(F.R, F.Hq + 2 * F.Hkv), dim3(64), 0, st, qj)) != cudaSuccess) return e;
    if (F.n_tok > 0) {
      AttnJob aj;
      aj.layer = i;
      aj.Hq = F.Hq;
      aj.Hkv = F.Hkv;
      aj.G = G;
      aj.R = F.R;
      aj.Rp = L.Rp;
      aj.GRp = G * L.Rp;
      aj.halves = L.halves;
      aj.n_tok = F.n_tok;
      aj.chunks = L.chunks;
      aj.q = q;
      aj.opart = opart;
      aj.mlpart = ml;
      aj.status = status;
      if ((e = launch_pdl(k_fw_attn, dim3(L.chunks, L.halves, F.Hkv), dim3(kAtThreads), kAtSmem, st,
                          km, vm, aj)) != cudaSuccess)
        return e;
    }
    AttnOutJob oj;
    oj.Hq = F.Hq;
    oj.Hkv = F.Hkv;
    oj.G = G;
    oj.R = F.R;
    oj.Rp = L.Rp;
    oj.halves = L.halves;
    oj.chunks = F.n_tok > 0 ? L.chunks : 0;
    oj.q = q;
    oj.k = kown;
    oj.v = vown;
    oj.opart = opart;
    oj.mlpart = ml;
    oj.o = X;
    oj.status = status;
    if ((e = launch_pdl(k_fw_attn_out, dim3(L.Rp * F.Hq), dim3(256), 0, st, oj)) != cudaSuccess)
      return e;
    if ((e = gemm(W.wo, D, D, X, F.R, L.Rp, L.sp_o, part, status, st)) != cudaSuccess) return e;
    // H += o Wo^T; X = bf16(RMSNorm(H) * ln2)
    nj.h_in = nullptr;
    nj.part = part;
    nj.splits = L.sp_o;
    nj.w = static_cast<const __nv_bfloat16*>(W.ln2);
    if ((e = norm(nj)) != cudaSuccess) return e;
    if (L.sp_gu == 1 && F.I % 64 == 0) {
      // one split: the SwiGLU product straight from the gate/up GEMM's epilogue
      if ((e = gemm(W.wgu, 2 * F.I, D, X, F.R, L.Rp, 1, part, status, st, F.I, Ab)) != cudaSuccess)
        return e;
    } else {
      if ((e = gemm(W.wgu, 2 * F.I, D, X, F.R, L.Rp, L.sp_gu, part, status, st)) != cudaSuccess) return e;
      SwigluJob sj;
      sj.part = part;
      sj.splits = L.sp_gu;
      sj.Rp = L.Rp;
      sj.R = F.R;
      sj.I = F.I;
      sj.A = Ab;
      if ((e = launch_pdl(k_fw_swiglu, dim3((unsigned)(((int64_t)L.Rp * F.I + 255) / 256)), dim3(256), 0, st, sj)) != cudaSuccess)
        return e;
    }
    if ((e = gemm(W.wd, D, F.I, Ab, F.R, L.Rp, L.sp_d, part, status, st)) != cudaSuccess) return e;
  }
  // H += the last down projection
  nj.h_in = nullptr;
  nj.part = part;
  nj.splits = L.sp_d;
  nj.w = nullptr;
  if ((e = norm(nj)) != cudaSuccess) return e;
  if (A.h_out)
    return cudaMemcpyAsync(A.h_out, H, (size_t)F.R * D * sizeof(float), cudaMemcpyDeviceToDevice, st);
  return cudaSuccess;
}

}  // namespace ss
