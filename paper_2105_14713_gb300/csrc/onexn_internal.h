// Internal helpers shared by the host and CUDA translation units of libonexn.
#pragma once

#include <stdint.h>

#include "onexn.h"

namespace onexn {

// Record a printf-style message for onexn_last_error() and return st.
onexn_status fail(onexn_status st, const char *fmt, ...);
void clear_error();
const char *last_error();
uint16_t bf16_bits_rne(float f);

}  // namespace onexn
