// Host-side descriptor validation and fp64 construction of the SDQ tables.
//
// The tables are the linear maps of Algorithm 1 (SDQ-LLM, arXiv 2510.03275)
// written as matrices:
//   encode   x_up = Resample(w . Had, n_b) = A_enc w,   A_enc = U Had^T
//   decode   W_hat_blk . x_b = alpha * c . (G x_b),     G = D^T Had^T
// U (n_b x B) is the band-limited upsampler of the Resample function: the
// B lowest frequencies kept, the Nyquist bin split half-and-half.  D^T
// (n_b x B) is the transpose of the downsampler n_b -> B: the same band, the
// two Nyquist aliases folded into one bin.  Both are evaluated here from
// their trigonometric-sum closed forms (not by FFT), with the cosine
// argument reduced exactly in integers: tau = (j B - k n_b) / (n_b B).
// Had = diag(d) H_B / sqrt(B) with H_B the Sylvester matrix of eq. (13), so
// (M Had^T)[j][k] = d_k / sqrt(B) * (H_B M[j])[k], applied with a fast
// Walsh-Hadamard transform.  Everything is fp64, rounded to fp32 once.
#include <cmath>
#include <cstring>
#include <vector>

#include "sdq_internal.h"

namespace sdq {

int validate(const sdq_layer_desc* d, Geometry* g) {
  if (!d) return SDQ_ERR_INVALID_ARG;
  const int64_t B = d->block;
  if (B < 2 || B > 1024 || (B & (B - 1))) return SDQ_ERR_INVALID_ARG;
  if (d->n_out < 1 || d->n_out > (1 << 24)) return SDQ_ERR_INVALID_ARG;
  if (d->k_in < 1 || d->k_in % B) return SDQ_ERR_INVALID_ARG;
  if (d->osr_den < 1 || d->osr_num < d->osr_den) return SDQ_ERR_INVALID_ARG;
  if ((B * d->osr_num) % d->osr_den) return SDQ_ERR_INVALID_ARG;
  const int64_t n_b = B * d->osr_num / d->osr_den;
  if (n_b > 4096) return SDQ_ERR_INVALID_ARG;
  if (d->quantizer != SDQ_BINARY && d->quantizer != SDQ_TERNARY) return SDQ_ERR_INVALID_ARG;
  if (d->hadamard != 0 && d->hadamard != 1) return SDQ_ERR_INVALID_ARG;
  if (d->alpha_mode != SDQ_ALPHA_MAXABS && d->alpha_mode != SDQ_ALPHA_MEANABS)
    return SDQ_ERR_INVALID_ARG;
  const int64_t nblk = d->k_in / B;
  const int64_t k_eff = nblk * n_b;
  if (k_eff > (int64_t(1) << 24)) return SDQ_ERR_INVALID_ARG;
  if (g) {
    g->n_out = d->n_out;
    g->k_in = d->k_in;
    g->block = (int32_t)B;
    g->n_b = (int32_t)n_b;
    g->nblk = (int32_t)nblk;
    g->k_eff = k_eff;
    g->bits = d->quantizer;
    g->words_per_row = (int32_t)(4 * ((k_eff * g->bits + 127) / 128));
    g->ntiles = (d->n_out + kTileRows - 1) / kTileRows;
    g->k_eff_pad = (k_eff + 127) / 128 * 128;
    g->ngroups = (int32_t)(g->k_eff_pad / kGroupCodes);
    g->wpg = kGroupCodes * g->bits / 32;
  }
  return SDQ_OK;
}

namespace {

// In-place fast Walsh-Hadamard transform (natural / Sylvester order):
// v <- H_n v with H_n[k][k'] = (-1)^popcount(k & k').
void fwht(double* v, int n) {
  for (int h = 1; h < n; h <<= 1)
    for (int i = 0; i < n; i += 2 * h)
      for (int k = i; k < i + h; ++k) {
        const double a = v[k], b = v[k + h];
        v[k] = a + b;
        v[k + h] = a - b;
      }
}

}  // namespace

int build_tables(const sdq_layer_desc* desc, const int8_t* signs, float* a_enc, float* gout, double* dt_out,
                 float* g_gptq) {
  Geometry g;
  int st = validate(desc, &g);
  if (st != SDQ_OK) return st;
  const int B = g.block, nb = g.n_b;
  std::vector<double> d(B, 1.0);
  if (signs) {
    for (int k = 0; k < B; ++k) {
      if (signs[k] != 1 && signs[k] != -1) return SDQ_ERR_INVALID_ARG;
      d[k] = signs[k];
    }
  }
  const bool had = desc->hadamard != 0;
  const double inv_sqrt_b = 1.0 / std::sqrt((double)B);

  // Upsampler U and downsampler transpose Dt, both n_b x B.
  std::vector<double> U((size_t)nb * B), Dt((size_t)nb * B);
  if (nb == B) {
    for (int j = 0; j < nb; ++j)
      for (int k = 0; k < B; ++k) U[(size_t)j * B + k] = Dt[(size_t)j * B + k] = (j == k);
  } else {
    // cos(2 pi i / P) for i in [0, P), P = n_b * B: every cosine below has an
    // argument that is an exact integer multiple of 2 pi / P.
    const int64_t P = (int64_t)nb * B;
    std::vector<double> ct((size_t)P);
    for (int64_t i = 0; i < P; ++i) ct[(size_t)i] = std::cos(2.0 * M_PI * (double)i / (double)P);
    auto cosP = [&](int64_t num) {  // cos(2 pi num / P)
      int64_t r = num % P;
      if (r < 0) r += P;
      return ct[(size_t)r];
    };
    const int half = B / 2;
    for (int j = 0; j < nb; ++j) {
      // Nyquist alias of the downsampler: 2 cos(pi B j / n_b) = 2 cos(2 pi (B/2) j B / P).
      const double nyq_d = 2.0 * cosP((int64_t)half * j * B);
      for (int k = 0; k < B; ++k) {
        const int64_t r = (int64_t)j * B - (int64_t)k * nb;  // tau = r / P
        double s = 0.0;
        for (int f = 1; f < half; ++f) s += cosP((int64_t)f * r);
        const double core = 1.0 + 2.0 * s;
        // Upsampler: split Nyquist bin, cos(pi B tau) = cos(2 pi (B/2) r / P).
        U[(size_t)j * B + k] = (core + cosP((int64_t)half * r)) / (double)B;
        Dt[(size_t)j * B + k] = (core + nyq_d * ((k & 1) ? -1.0 : 1.0)) / (double)nb;
      }
    }
  }
  if (dt_out) std::memcpy(dt_out, Dt.data(), sizeof(double) * Dt.size());
  // Right-multiply by Had^T: row j -> d_k / sqrt(B) * (H_B row_j)[k].
  std::vector<double> row(B);
  for (int which = 0; which < 2; ++which) {
    std::vector<double>& M = which ? Dt : U;
    float* out = which ? gout : a_enc;
    if (!out && !(which && g_gptq)) continue;
    for (int j = 0; j < nb; ++j) {
      std::memcpy(row.data(), &M[(size_t)j * B], sizeof(double) * B);
      if (had) {
        fwht(row.data(), B);
        for (int k = 0; k < B; ++k) row[k] *= d[k] * inv_sqrt_b;
      }
      // Entries that are exactly zero in real arithmetic (interpolation nodes
      // at integer OSR, Hadamard cancellations) carry fp64 noise of ~1e-16;
      // they are set to exact zero, below 2^-46, before rounding to fp32.
      if (out)
        for (int k = 0; k < B; ++k)
          out[(size_t)j * B + k] = std::fabs(row[k]) < 0x1p-46 ? 0.0f : (float)row[k];
      // G of the GPTQ block reconstruction: rounded to the nearest multiple of
      // 2^-30 (ties to even) before fp32, so that fp64 errors of entries that
      // come out of cancellations cannot change their fp32 value
      if (which && g_gptq)
        for (int k = 0; k < B; ++k) g_gptq[(size_t)j * B + k] = (float)(std::nearbyint(row[k] * 0x1p30) * 0x1p-30);
    }
  }
  return SDQ_OK;
}

}  // namespace sdq

extern "C" int sdq_build_tables(const sdq_layer_desc* desc, const int8_t* had_signs,
                                float* a_enc_host, float* g_host) {
  return sdq::build_tables(desc, had_signs, a_enc_host, g_host);
}

extern "C" int sdq_build_gptq_table(const sdq_layer_desc* desc, const int8_t* had_signs, float* g_host) {
  if (!g_host) return SDQ_ERR_INVALID_ARG;
  return sdq::build_tables(desc, had_signs, nullptr, nullptr, nullptr, g_host);
}

extern "C" int64_t sdq_k_eff(const sdq_layer_desc* desc) {
  sdq::Geometry g;
  return sdq::validate(desc, &g) == SDQ_OK ? g.k_eff : 0;
}

extern "C" size_t sdq_plain_bytes(const sdq_layer_desc* desc) {
  sdq::Geometry g;
  if (sdq::validate(desc, &g) != SDQ_OK) return 0;
  return (size_t)g.n_out * g.words_per_row * 4;
}

extern "C" size_t sdq_tiled_bytes(const sdq_layer_desc* desc) {
  sdq::Geometry g;
  if (sdq::validate(desc, &g) != SDQ_OK) return 0;
  return (size_t)g.ntiles * g.ngroups * sdq::kTileRows * g.wpg * 4;
}

extern "C" const char* sdq_status_string(int s) {
  switch (s) {
    case SDQ_OK: return "SDQ_OK";
    case SDQ_ERR_INVALID_ARG: return "SDQ_ERR_INVALID_ARG: invalid argument";
    case SDQ_ERR_UNSUPPORTED: return "SDQ_ERR_UNSUPPORTED: unsupported configuration or device";
    case SDQ_ERR_WORKSPACE: return "SDQ_ERR_WORKSPACE: workspace too small";
    case SDQ_ERR_CUDA: return "SDQ_ERR_CUDA: CUDA runtime error";
    case SDQ_ERR_TIMEOUT: return "SDQ_ERR_TIMEOUT: bounded device wait expired";
    case SDQ_ERR_BAD_CODE: return "SDQ_ERR_BAD_CODE: invalid ternary code pattern";
    case SDQ_ERR_ALLOC: return "SDQ_ERR_ALLOC: allocation failed";
    default: return "unknown sdq status";
  }
}
