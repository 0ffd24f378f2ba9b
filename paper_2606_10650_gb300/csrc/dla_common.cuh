// dla_common.cuh -- shared device helpers of the DLA sm_103a kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "dla_kernels.h"
#include "dla_sm100.cuh"

namespace dla {

// State Information Score from three scalars of the token state s = v k^T
// and the open state S (Sec. 3.1 / Algorithm 1 with the whole-matrix RMSNorm
// N(X) = X / sqrt(||X||^2 / D + rms_eps)):
//   a = ||s||^2 = ||k||^2 ||v||^2,  beta = <s, S> = v^T S k,  gam = ||S||^2.
// Mode 0 compares N(s) with N(S) (Algorithm 1); mode 1 compares N(S + s)
// with N(S) (Eq. importance_score read literally).  With x = ||N(A)||,
// y = ||N(B)|| and c = <A,B> / (||A|| ||B||),
//   ||N(A) - N(B)||^2 = (x - y)^2 + 2 x y (1 - c),
// a form without the cancellation of x^2 + y^2 - 2xyc; it needs no d x d work
// once a, beta, gam are known.  Evaluated in fp32 (GB300's fp64 rate is a
// small fraction of its fp32 rate); the inputs carry ~1e-7 relative error.
__device__ __forceinline__ float info_score(float a, float beta, float gam, float D, const ScoreParams& p) {
  float AA, BB, AB;
  if (p.score_mode == 1) {
    AA = gam + 2.f * beta + a;
    BB = gam;
    AB = gam + beta;
  } else {
    AA = a;
    BB = gam;
    AB = beta;
  }
  AA = fmaxf(AA, 0.f);
  BB = fmaxf(BB, 0.f);
  const float re = (float)p.rms_eps;
  const float x = sqrtf(AA / (AA / D + re));
  const float y = sqrtf(BB / (BB / D + re));
  const float nab = sqrtf(AA) * sqrtf(BB);
  const float c = nab > 0.f ? fminf(fmaxf(AB / nab, -1.f), 1.f) : 0.f;
  const float num2 = (x - y) * (x - y) + 2.f * x * y * (1.f - c);
  return sqrtf(fmaxf(num2, 0.f)) / (y + (float)p.eps);
}

// The same score as info_score, from hardware reciprocal square roots and an
// approximate divide (a few ulp; invD = 1 / D).  For the latency-bound
// boundary passes of the scan: each pass waits on one score per token.
__device__ __forceinline__ float info_score_fast(float a, float beta, float gam, float invD, const ScoreParams& p) {
  float AA, BB, AB;
  if (p.score_mode == 1) {
    AA = gam + 2.f * beta + a;
    BB = gam;
    AB = gam + beta;
  } else {
    AA = a;
    BB = gam;
    AB = beta;
  }
  AA = fmaxf(AA, 0.f);
  BB = fmaxf(BB, 0.f);
  const float re = p.rms_eps_f;
  const float rA = rsqrtf(AA), rB = rsqrtf(BB);
  const float sA = rsqrtf(fmaf(AA, invD, re)), sB = rsqrtf(fmaf(BB, invD, re));
  // |N(A)| = sqrt(AA) / sqrt(AA / D + re), likewise for B; c = <A, B> / (|A| |B|)
  const float x = (AA > 0.f) ? AA * rA * sA : 0.f;
  const float y = (BB > 0.f) ? BB * rB * sB : 0.f;
  const float c = (AA > 0.f && BB > 0.f) ? fminf(fmaxf(AB * rA * rB, -1.f), 1.f) : 0.f;
  const float num2 = fmaxf((x - y) * (x - y) + 2.f * x * y * (1.f - c), 0.f);
  const float nrm = (num2 > 0.f) ? num2 * rsqrtf(num2) : 0.f;
  return __fdividef(nrm, y + p.eps_f);
}

// ---- flags shared with a concurrently running kernel
__device__ __forceinline__ int ld_acquire_gpu(const int32_t* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_gpu(int32_t* p, int v) {
  asm volatile("st.release.gpu.global.b32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
// This stream's end of the round [t_begin, t_end): the call's t_end, or, with
// per-row lengths, row b's length clamped to [t_begin, t_end] (tokens past it
// are padding).
__device__ __forceinline__ int row_t_end(const int32_t* seq_lens, int b, int t_begin, int t_end) {
  if (!seq_lens) return t_end;
  return max(t_begin, min(t_end, __ldg(seq_lens + b)));
}
// fp16 pool entries: an entry holds S / s in fp16, s a power of two chosen from
// an upper bound of |S|_F (f16_scale), so that no element exceeds 2^13 (eight
// times below the fp16 range) and every element keeps fp16's 2^-12 relative
// rounding.  The bounds come from the triangle inequality over exact norms, so
// the range needs no check per element.
__device__ __forceinline__ float f16_scale(float bound) {
  if (!(bound > 0.f) || !isfinite(bound)) return 1.f;  // an infinite state is caught by the range check
  int ex;
  frexpf(bound, &ex);               // bound < 2^ex
  return ldexpf(1.f, ex - 13);      // bound / s < 2^13
}
__device__ __forceinline__ uint2 f16x4(float4 x, float inv) {
  const __half2 a = __floats2half2_rn(x.x * inv, x.y * inv), b = __floats2half2_rn(x.z * inv, x.w * inv);
  return make_uint2(*reinterpret_cast<const uint32_t*>(&a), *reinterpret_cast<const uint32_t*>(&b));
}
// Token row of the first token of batch row b: b * T in the padded layout, or
// row_start[b] in the packed one.
__device__ __forceinline__ long long row_tok0(const int32_t* row_start, int b, int T) {
  return row_start ? (long long)__ldg(row_start + b) : (long long)b * T;
}
// Decision trace of padding tokens [t0, t1) of one stream: no boundary, no merge.
__device__ __forceinline__ void fill_padding_trace(uint8_t* bnd, int32_t* mlog, int t0, int t1, int i0, int ni) {
  for (int t = t0 + i0; t < t1; t += ni) {
    bnd[t] = 0;
    mlog[t] = -1;
  }
}

// Read-out side: thread 0 waits until the scan CTAs of stream bh have completed
// `need` intervals (progress[bh][0 .. ctas)), at most the wait limit (then
// status 5) and not once the status word reports a failure; the caller's CTA
// barrier then orders every later read after the wait.  Data the scan writes
// must then be read past L1 (__ldcg): another CTA on the SM may hold an older
// copy of the line.
__device__ __forceinline__ void wait_progress(const int32_t* progress, int ctas, int bh, int need, int32_t* status) {
  if (!progress || threadIdx.x != 0) return;
  const long long t0 = clock64();
  long long lim = -1;
  for (int r = 0; r < ctas; ++r)
    while (ld_acquire_gpu(progress + 2 * bh + r) < need) {
      if (*(volatile int32_t*)status != 0) return;  // the call has failed already
      if (sm100::wait_expired(t0, lim, status)) {
        atomicCAS(status, 0, sm100::kStatusTimeout);
        return;
      }
    }
}

template <typename T>
__device__ __forceinline__ float to_f32(T x);
template <>
__device__ __forceinline__ float to_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T>
__device__ __forceinline__ T from_f32(float x);
template <>
__device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

// Loads 4 consecutive elements (16-byte aligned for fp32, 8-byte for bf16) as floats.
__device__ __forceinline__ float4 load4(const float* p) { return *reinterpret_cast<const float4*>(p); }
__device__ __forceinline__ float4 load4(const __nv_bfloat16* p) {
  uint2 u = *reinterpret_cast<const uint2*>(p);
  __nv_bfloat162 a = *reinterpret_cast<__nv_bfloat162*>(&u.x);
  __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162*>(&u.y);
  float2 fa = __bfloat1622float2(a), fb = __bfloat1622float2(b);
  return make_float4(fa.x, fa.y, fb.x, fb.y);
}

__device__ __forceinline__ void store4(float* p, float4 v) { *reinterpret_cast<float4*>(p) = v; }
__device__ __forceinline__ void store4(__nv_bfloat16* p, float4 v) {
  __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y);
  __nv_bfloat162 b = __floats2bfloat162_rn(v.z, v.w);
  uint2 u;
  u.x = *reinterpret_cast<uint32_t*>(&a);
  u.y = *reinterpret_cast<uint32_t*>(&b);
  *reinterpret_cast<uint2*>(p) = u;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Cache metadata of the live entries, held in registers by one warp: entry i
// in lane i % 32, element i / 32 (C <= 64).  i is warp-uniform.
template <typename T>
__device__ __forceinline__ T entry_get(const T (&f)[2], int i) {
  return __shfl_sync(0xffffffffu, (i < 32) ? f[0] : f[1], i & 31);
}
template <typename T>
__device__ __forceinline__ void entry_set(T (&f)[2], int i, T v) {
  if ((i & 31) == (int)(threadIdx.x & 31)) {
    if (i < 32) f[0] = v;
    else f[1] = v;
  }
}
// Entry i + 1's field for both of this lane's entries (i = lane, lane + 32).
template <typename T>
__device__ __forceinline__ void entry_next(const T (&f)[2], T (&nx)[2]) {
  const int lane = threadIdx.x & 31;
  nx[0] = __shfl_sync(0xffffffffu, lane == 0 ? f[1] : f[0], (lane + 1) & 31);
  nx[1] = __shfl_down_sync(0xffffffffu, f[1], 1);
}

// Warp argmin over (value, index) pairs; lowest index wins exact ties.
__device__ __forceinline__ void warp_argmin(double& v, int& i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    double ov = __shfl_xor_sync(0xffffffffu, v, o);
    int oi = __shfl_xor_sync(0xffffffffu, i, o);
    if (ov < v || (ov == v && oi < i)) {
      v = ov;
      i = oi;
    }
  }
}

// Adjacent-pair argmin of Algorithm 2 over logical entries 0..m-1 (m >= 2):
// i* = argmin_i (Ibar_i + Ibar_{i+1}) / (n_i + n_{i+1}), lowest i on ties.
// Called by one full warp; every lane returns i*.
__device__ __forceinline__ int pair_argmin_warp(const int* n, const double* ibar, int m) {
  const int lane = threadIdx.x & 31;
  double best = 1.0 / 0.0;
  int bi = 0x7fffffff;
  for (int i = lane; i + 1 < m; i += 32) {
    double dens = (ibar[i] + ibar[i + 1]) / (double)(n[i] + n[i + 1]);
    if (dens < best) {
      best = dens;
      bi = i;
    }
  }
  warp_argmin(best, bi);
  return bi;
}

}  // namespace dla
