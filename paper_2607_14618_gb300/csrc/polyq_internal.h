// Internal declarations shared by the library's translation units.
#pragma once
#include <stdint.h>

#include "polyq.h"

int polyq_set_error(int code, const char* fmt, ...);
void polyq_clear_error();
int polyq_check_dev_layer(const polyq_dev_layer* L, const char* who);
