// headlogits.cuh — logits of G query heads against 32 consecutive key rows
// with the 2G-lanes-per-row geometry shared by the decode kernel and the
// evaluation kernels.
#pragma once

#include "common.cuh"

namespace certkv {

// Lane geometry of the logits for G query heads: 2G lanes share one slot, each
// holding 128 / 2G of the G queries' dimensions in registers, so every K row
// is read once, coalesced, and a transposing shuffle reduction leaves lane i of
// the slot's group with the logit of head i mod G.
template <int G>
struct DecGeo {
  static constexpr int LPS = 2 * G;           // lanes per slot
  static constexpr int SPP = 32 / LPS;        // slots per pass
  static constexpr int NP = 32 / SPP;        // passes per 32-token tile
  static constexpr int DPL = kD / LPS;        // dimensions per lane
  static constexpr int NPAIR = DPL / 2;       // fp32 pairs per lane and head
};

// v[h]: this lane's partial dot product for head h.  Returns the full dot
// product of head (lane mod G) over the 2G lanes of the slot group.
template <int G>
__device__ __forceinline__ float reduce_heads(float (&v)[G], int lane) {
#pragma unroll
  for (int o = G / 2; o >= 1; o >>= 1) {
    const bool upper = (lane & o) != 0;
#pragma unroll
    for (int k = 0; k < o; ++k) {
      const float keep = upper ? v[k + o] : v[k];
      const float send = upper ? v[k] : v[k + o];
      v[k] = keep + __shfl_xor_sync(kFull, send, o);
    }
  }
  return v[0] + __shfl_xor_sync(kFull, v[0], G);
}

// This lane's slice of the G query rows q_g (bf16 [G][kD], row g at q + g kD),
// as fp32 pairs in the order the key chunks are read.
template <int G>
__device__ __forceinline__ void load_query_slice(const __nv_bfloat16* __restrict__ q, int lane,
                                                 float2 (&qr)[DecGeo<G>::NPAIR][G]) {
  using Geo = DecGeo<G>;
  const int gi = lane % Geo::LPS;
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const uint32_t* qg = reinterpret_cast<const uint32_t*>(q + (size_t)g * kD);
#pragma unroll
    for (int j = 0; j < Geo::NPAIR; ++j) {
      const int dim = Geo::DPL >= 8 ? 8 * (gi + Geo::LPS * (j / 4)) + 2 * (j % 4)
                                    : Geo::DPL * gi + 2 * j;
      const uint32_t w = __ldg(qg + dim / 2);
      qr[j][g] = make_float2(bf16lo(w), bf16hi(w));
    }
  }
}

// Dot products of the G query rows with the key rows K[0 .. cnt) (bf16 rows of
// kD, global memory, 16-byte aligned) written to xs[row G + g] (shared memory,
// one warp's 32 x G floats); rows past cnt are not read.  The 2G lanes of a
// row group read the row's 16-byte chunks gi + LPS c, coalesced.
template <int G>
__device__ __forceinline__ void tile_head_logits(const __nv_bfloat16* __restrict__ K, int cnt,
                                                 const float2 (&qr)[DecGeo<G>::NPAIR][G], int lane,
                                                 float* __restrict__ xs) {
  using Geo = DecGeo<G>;
  const int gi = lane % Geo::LPS, gs = lane / Geo::LPS;
  float xl[Geo::NP];
#pragma unroll
  for (int ps = 0; ps < Geo::NP; ++ps) {
    const int row = ps * Geo::SPP + gs;
    const unsigned char* rp = reinterpret_cast<const unsigned char*>(K + (size_t)row * kD);
    float2 x2[G];
#pragma unroll
    for (int g = 0; g < G; ++g) x2[g] = make_float2(0.f, 0.f);
    if (row < cnt) {
      if constexpr (Geo::DPL >= 8) {
        uint4 raw[Geo::DPL / 8];
#pragma unroll
        for (int c = 0; c < Geo::DPL / 8; ++c)
          raw[c] = __ldg(reinterpret_cast<const uint4*>(rp + (gi + Geo::LPS * c) * 16));
#pragma unroll
        for (int c = 0; c < Geo::DPL / 8; ++c) {
          const float2 kp[4] = {make_float2(bf16lo(raw[c].x), bf16hi(raw[c].x)),
                                make_float2(bf16lo(raw[c].y), bf16hi(raw[c].y)),
                                make_float2(bf16lo(raw[c].z), bf16hi(raw[c].z)),
                                make_float2(bf16lo(raw[c].w), bf16hi(raw[c].w))};
#pragma unroll
          for (int e = 0; e < 4; ++e)
#pragma unroll
            for (int g = 0; g < G; ++g) x2[g] = ffma2(qr[4 * c + e][g], kp[e], x2[g]);
        }
      } else {
        const uint2 raw = __ldg(reinterpret_cast<const uint2*>(rp + gi * 8));
        const float2 kp[2] = {make_float2(bf16lo(raw.x), bf16hi(raw.x)),
                              make_float2(bf16lo(raw.y), bf16hi(raw.y))};
#pragma unroll
        for (int e = 0; e < 2; ++e)
#pragma unroll
          for (int g = 0; g < G; ++g) x2[g] = ffma2(qr[e][g], kp[e], x2[g]);
      }
    }
    float v[G];
#pragma unroll
    for (int g = 0; g < G; ++g) v[g] = x2[g].x + x2[g].y;
    xl[ps] = reduce_heads<G>(v, lane);
  }
  if (gi < G) {
#pragma unroll
    for (int ps = 0; ps < Geo::NP; ++ps) xs[(ps * Geo::SPP + gs) * G + gi] = xl[ps];
  }
  __syncwarp();
}

}  // namespace certkv
