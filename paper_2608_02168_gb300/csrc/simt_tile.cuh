// CUDA-core (fp32 FMA) tile helpers shared by the projection and alignment kernels.
// A block of 256 threads owns a 64-row tile; thread (ty, tx) = (tid / 16, tid % 16) holds rows
// ty*RM .. ty*RM+RM-1 and the contiguous columns tx*CN .. tx*CN+CN-1, so the 16 threads of a row
// form one half-warp and row reductions are 16-lane shuffles.
#pragma once

#include "hg_internal.cuh"

namespace hg {

constexpr int kBM = 64;       // rows per block
constexpr int kKC = 32;       // K chunk
constexpr int kAPad = kKC + 4;

__device__ __forceinline__ float act_apply(float u, int act) {
  if (act == HG_ACT_RELU) return u > 0.f ? u : 0.f;
  if (act == HG_ACT_GELU_TANH) {
    const float k = 0.7978845608028654f;
    return 0.5f * u * (1.f + tanhf(k * (u + 0.044715f * u * u * u)));
  }
  return u;
}

__device__ __forceinline__ float act_grad(float u, int act) {
  if (act == HG_ACT_RELU) return u > 0.f ? 1.f : 0.f;
  if (act == HG_ACT_GELU_TANH) {
    const float k = 0.7978845608028654f;
    const float t = tanhf(k * (u + 0.044715f * u * u * u));
    return 0.5f * (1.f + t) + 0.5f * u * (1.f - t * t) * k * (1.f + 3.f * 0.044715f * u * u);
  }
  return 1.f;
}

template <typename T, int D>
struct Tile {
  static constexpr int CN = D / 16;  // columns per thread (contiguous)
  static constexpr int RM = kBM / 16;  // rows per thread (ty * RM + i)
  static constexpr int kVec = VecTraits<T>::kElems;
};

// Stage A[m][k0 .. k0+KC) for rows a_row0 + m (m < kBM, zero past n_valid) into As (fp32).  With
// a row map, row a_row0 + m of A is A[map[a_row0 + m]], and a mapped index >= sentinel is a zero row.
template <typename T, int D>
__device__ __forceinline__ void stage_a(float (*As)[kAPad], const T* __restrict__ A, int64_t a_row0, int64_t n_valid,
                                        int k0, const int32_t* __restrict__ map = nullptr, int64_t sentinel = 0) {
  constexpr int VEC = VecTraits<T>::kElems;
  constexpr int PER_ROW = kKC / VEC;
  for (int idx = threadIdx.x; idx < kBM * PER_ROW; idx += blockDim.x) {
    const int m = idx / PER_ROW, kv = idx % PER_ROW;
    float f[VEC];
    const int64_t row = m < n_valid ? (map ? (int64_t)map[a_row0 + m] : a_row0 + m) : 0;
    if (m < n_valid && (!map || row < sentinel)) {
      unpack(ldg16(A + row * D + k0 + kv * VEC), f, T());
    } else {
#pragma unroll
      for (int q = 0; q < VEC; ++q) f[q] = 0.f;
    }
#pragma unroll
    for (int q = 0; q < VEC; ++q) As[m][kv * VEC + q] = f[q];
  }
}

// Stage rows k0 .. k0+KC of a D x D row-major matrix B into Bs (fp32).
template <typename T, int D>
__device__ __forceinline__ void stage_b(float* Bs, const T* __restrict__ B, int k0) {
  constexpr int VEC = VecTraits<T>::kElems;
  for (int idx = threadIdx.x; idx < kKC * D / VEC; idx += blockDim.x) {
    const int k = idx / (D / VEC), nv = idx % (D / VEC);
    float f[VEC];
    unpack(ldg16(B + (int64_t)(k0 + k) * D + nv * VEC), f, T());
#pragma unroll
    for (int q = 0; q < VEC; ++q) Bs[k * D + nv * VEC + q] = f[q];
  }
}

// acc[i][j] += sum_k A(ty*RM+i, k) * Bs[k][tx*CN + j] for k in [0, KC), A from an fp32 smem tile
// with row stride lda and column offset kofs.
template <int D, int RM, int CN>
__device__ __forceinline__ void mma_chunk(const float* A, int lda, int kofs, const float* Bs, float (&acc)[RM][CN]) {
  const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
#pragma unroll 4
  for (int k = 0; k < kKC; ++k) {
    float a[RM];
#pragma unroll
    for (int i = 0; i < RM; ++i) a[i] = A[(ty * RM + i) * lda + kofs + k];
    float b[CN];
#pragma unroll
    for (int j = 0; j < CN; j += 4) {
      float4 v = *reinterpret_cast<const float4*>(Bs + k * D + tx * CN + j);
      b[j] = v.x;
      b[j + 1] = v.y;
      b[j + 2] = v.z;
      b[j + 3] = v.w;
    }
#pragma unroll
    for (int i = 0; i < RM; ++i)
#pragma unroll
      for (int j = 0; j < CN; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
  }
}

// Sum of v over the 16 lanes that share a row (one half-warp).
__device__ __forceinline__ float row_sum16(float v) {
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename T, int CN>
__device__ __forceinline__ void load_cols(const T* __restrict__ p, float* out) {
  constexpr int VEC = VecTraits<T>::kElems;
#pragma unroll
  for (int j = 0; j < CN; j += VEC) {
    if constexpr (CN >= VEC) {
      unpack(ldg16(p + j), out + j, T());
    }
  }
  if constexpr (CN < VEC) {
#pragma unroll
    for (int j = 0; j < CN; ++j) out[j] = to_f32(p[j]);
  }
}

template <typename T, int CN>
__device__ __forceinline__ void store_cols(T* __restrict__ p, const float* v) {
  constexpr int VEC = VecTraits<T>::kElems;
  if constexpr (CN >= VEC) {
#pragma unroll
    for (int j = 0; j < CN; j += VEC) st16(p + j, pack(v + j, T()));
  } else {
#pragma unroll
    for (int j = 0; j < CN; ++j) p[j] = from_f32<T>(v[j]);
  }
}

template <typename T>
__device__ __forceinline__ float round_to(float x) {
  return to_f32(from_f32<T>(x));
}

}  // namespace hg
