/* Host (CPU) twin of synth/gen.py: the same bf16 bytes as the numpy
 * generator, for hidden-state rows and K/V rows, written in plain C so that
 * the oracle's inputs at full size (tens of thousands of 32-layer rows) take
 * seconds instead of minutes.  It holds none of the eviction method's
 * arithmetic.  Every float operation is a separate rounded float32 operation
 * (built with -ffp-contract=off, so no fused multiply-add can change a bit
 * relative to numpy), and the integer hash is the SplitMix64 output function
 * (Steele, Lea and Flood, OOPSLA 2014).  Plain C99, no intrinsics: it gives
 * the same bytes on x86-64 and aarch64. */
#include <stdint.h>
#include <string.h>

#define GAMMA 0x9E3779B97F4A7C15ull
#define MUL1 0xBF58476D1CE4E5B9ull
#define MUL2 0x94D049BB133111EBull
#define S_HIDDEN 1u
#define S_SEGMENT 2u
#define S_KEY 4u
#define S_VALUE 5u

static inline uint64_t mix64(uint64_t x) {
  uint64_t z = x + GAMMA;
  z = (z ^ (z >> 30)) * MUL1;
  z = (z ^ (z >> 27)) * MUL2;
  return z ^ (z >> 31);
}

static inline uint64_t row_key(uint64_t stream, uint64_t seed, uint64_t seq, uint64_t layer, uint64_t head,
                               uint64_t pos) {
  uint64_t k = mix64(mix64(seed) ^ stream);
  k = mix64(k ^ seq);
  k = mix64(k ^ ((layer << 16) | head));
  return mix64(k ^ pos);
}

/* Irwin-Hall sum of the four 16-bit lanes, centred: an exact integer, exact in float32. */
static inline float normal16(uint64_t e) {
  const int32_t s = (int32_t)(e & 0xFFFFu) + (int32_t)((e >> 16) & 0xFFFFu) + (int32_t)((e >> 32) & 0xFFFFu) +
                    (int32_t)(e >> 48);
  return (float)(s - 131070);
}

/* float32 -> bf16 bits, round to nearest even (finite inputs). */
static inline uint16_t bf16_rne(float v) {
  uint32_t b;
  memcpy(&b, &v, 4);
  const uint32_t r = ((b >> 16) & 1u) + 0x7FFFu;
  return (uint16_t)((b + r) >> 16);
}

/* Rows [n][D] of hidden layer `layer` of sequence `seq` at positions pos[i];
 * seg[i] is the Band A segment index of pos[i] (ignored when seg_amp == 0). */
int synth_host_hidden(uint64_t seed, int seq, int layer, const int64_t* pos, int64_t n, int D, float scale,
                      float drift, float seg_amp, float inv_sd, const float* mean, const int32_t* seg,
                      uint16_t* out) {
  if (n < 0 || D < 1 || !pos || !mean || !out || (seg_amp != 0.0f && !seg)) return 1;
  const float two_m16 = 1.52587890625e-05f; /* 2^-16 */
  const float bamp = seg_amp * inv_sd;
  for (int64_t i = 0; i < n; ++i) {
    const uint64_t key = row_key(S_HIDDEN, seed, (uint64_t)seq, (uint64_t)layer, 0, (uint64_t)pos[i]);
    const float tf = (float)pos[i] * two_m16;
    const float dt = drift * tf;
    const float one_dt = 1.0f + dt;
    const float sc = scale * one_dt;
    const float c = sc * inv_sd;
    const uint64_t skey =
        seg_amp != 0.0f ? row_key(S_SEGMENT, seed, (uint64_t)seq, (uint64_t)layer, 0, (uint64_t)seg[i]) : 0;
    uint16_t* row = out + i * (int64_t)D;
    for (int j = 0; j < D; ++j) {
      float v = normal16(mix64(key + (uint64_t)j)) * c;
      if (seg_amp != 0.0f) {
        const float y = normal16(mix64(skey + (uint64_t)j)) * bamp;
        v = v + y;
      }
      v = v + mean[j];
      row[j] = bf16_rne(v);
    }
  }
  return 0;
}

/* Rows [n][L][H][d] of the keys (kind 0) or values (kind 1) of sequence `seq`
 * at positions pos[i]; spike[i] != 0 marks a spike position (amplitude x4).
 * kv_scale: [L][H] of this kind; kv_off: [L][H][d] of this kind. */
int synth_host_kv(uint64_t seed, int seq, int kind, const int64_t* pos, const uint8_t* spike, int64_t n, int L,
                  int H, int d, const float* kv_scale, const float* kv_off, uint16_t* out) {
  if (n < 0 || L < 1 || H < 1 || d < 1 || !pos || !spike || !kv_scale || !kv_off || !out) return 1;
  const uint64_t stream = kind == 0 ? S_KEY : S_VALUE;
  for (int64_t i = 0; i < n; ++i) {
    const float amp = spike[i] ? 4.0f : 1.0f;
    for (int l = 0; l < L; ++l)
      for (int h = 0; h < H; ++h) {
        const uint64_t key = row_key(stream, seed, (uint64_t)seq, (uint64_t)l, (uint64_t)h, (uint64_t)pos[i]);
        const float cs = kv_scale[l * H + h] * amp;
        const float* off = kv_off + ((int64_t)l * H + h) * d;
        uint16_t* row = out + (((i * L) + l) * (int64_t)H + h) * d;
        for (int j = 0; j < d; ++j) {
          const float x = normal16(mix64(key + (uint64_t)j)) * cs;
          row[j] = bf16_rne(x + off[j]);
        }
      }
  }
  return 0;
}
